"""CPU oracle of the budget-conditioned gated prefill (test infrastructure only)."""
