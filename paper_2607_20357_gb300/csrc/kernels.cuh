// Declarations of the non-GEMM kernels and their launchers.
#pragma once

#include "common.cuh"

namespace svl {

constexpr int kSelectThreads = 512;
constexpr int kAttnQ = 256;       // query rows per attention work item (the kernel runs its two 128-row halves as units)
// n-tiles per raster band of the residual GEMMs' tile lists (O, down). A band
// sweeps all m-tiles while its weight columns stay in L2, so the input rows
// are read once per band: wider bands read them fewer times until the band's
// weights (band x 256 rows x K) no longer stay in L2 (about 45 MB).
constexpr int kNBand = 8;         // down list (16 n-tiles of 256 x 11,008 weights)
constexpr int kNBandO = 16;       // O list (16 n-tiles of 256 x 4,096 weights: one band)
// The N-sparse lists (QKV, gate/up) run in bands of m-tiles whose input rows
// total at most this many bytes: a band sweeps all n-tiles while its rows
// stay in L2, so the rows are read once and the weights once per band. At
// LLaVA-7B widths and b = 1 the 84 MB of rows make two bands (gate/up: 0.71
// GB of DRAM traffic per launch, against 0.87 GB in bands of 20 n-tiles and
// 0.84 GB with 27 MB of rows per band); a batch whose rows fit in one band
// reads everything once. 100 MB of rows in one band no longer stay in L2
// (4.2 GB).
constexpr long long kMBandBytes = 40ll << 20;
constexpr int kBM_SCHED = 128;    // tile rows (the GEMM's M)

struct SelectArgs {
  const float* scores;
  const int* vis_off;
  const int* text_len;
  const float* budget;
  const int* keep_count;
  const uint8_t* layer_gate;
  const uint8_t* group_gate;
  int L, G, P;
  long long D, Dkv, Di, V;
  int* k_out;
  uint32_t* flags;
  int* kept_local;
  // the paper's own rule (Sec. 3.1, 3.3): gates from compute-controller
  // logits (> 0), k = min(#{z > 0}, budget count), group fallback; nullptr:
  // gates given, k = budget count
  const float* gate_logits;  // [B, L, G]
  uint8_t* layer_gate_out;   // [B, L] projected gates (paper rule)
  uint8_t* group_gate_out;   // [B, L, G]
  int threshold_only;        // paper rule, gates decided later: k = #{z > 0}
  float* kappa;              // [B] sum sigma(z) / N, or nullptr
};

void launch_budget_embed(const float* budget, const __nv_bfloat16* w1, const __nv_bfloat16* w2, int H, int B,
                         float* e_b, cudaStream_t s);
void launch_select(const SelectArgs& a, int B, cudaStream_t s);
void launch_compact(int B, const int* vis_off, const int* k, const int* kept_local, int* kept_idx, int* kept_off,
                    int* kept_total, cudaStream_t s);

// ---------------------------------------------------------------- pack
struct PackArgs {
  int B, D, c_vis, V;
  int t_cap;
  const __nv_bfloat16* vis;
  const int* vis_off;
  const int* kept_idx;
  const int* kept_off;
  const int* text_ids;
  const int* text_off;
  const __nv_bfloat16* embed;
  __nv_bfloat16* X;
  int* cu_seqlens;
  int* pos;
  int* t_total;            // device scalar: T
  int use_projector;       // 1: visual rows go to the staging buffer
  __nv_bfloat16* stage;    // [kept_total, c_vis]
  int* row_map;            // [kept_total] -> row of X
  const __nv_bfloat16* tok_rows;  // [B, D] budget-token rows appended after the text, or nullptr
  uint32_t* status;
};
// e^LLM_b = W2 SiLU(W1 PE(b)) (Sec. 3.2: the Eq. 5 encoding, its own MLP to D), bf16 rows.
void launch_llm_budget_embed(const float* budget, const __nv_bfloat16* w1, const __nv_bfloat16* w2, int H, int D,
                             int B, __nv_bfloat16* out, cudaStream_t s);
void launch_pack_offsets(const PackArgs& a, cudaStream_t s);
void launch_offsets_diff(const int* off, int* len, int B, cudaStream_t s);
void launch_pack_gather(const PackArgs& a, cudaStream_t s);

// Sample b of the packed row r: cu[b] <= r < cu[b+1].
SVL_DEVINL int find_sample(const int* cu, int B, int r) {
  int lo = 0, hi = B;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (cu[mid] <= r) lo = mid; else hi = mid;
  }
  return lo;
}

// ---------------------------------------------------------------- e4m3 operands
// Per-row e4m3 quantisation of bf16 rows (times a gain vector when given:
// the input norm's gain of the QKV and gate/up projections). Row r of src holds G groups of kg
// columns; dst row r holds G groups of kgp >= kg codes (the tail of each
// group zero, so that every group starts on a 128-byte K block). Only the
// groups active for the row's sample are read and quantised (the others are
// written as zeros): gates of layer l when group_gate is given, else all.
// Rows at or past cu_seqlens[B] (when given) are left untouched.
struct QuantArgs {
  const __nv_bfloat16* src;
  const __nv_bfloat16* gain;  // [G * kg] multiplies each row before quantising, or nullptr
  int64_t ld_src;
  int64_t rows;
  int G, kg, kgp;
  uint8_t* dst;
  int64_t ld_dst;
  float* scale;  // [rows]: amax / 448 (0 for a row without a non-zero value)
  const int* cu_seqlens;
  int B;
  const uint8_t* layer_gate;  // [B, L] or nullptr
  const uint8_t* group_gate;  // [B, L, G] or nullptr
  int L, l, P;
};
cudaError_t launch_quant_rows(const QuantArgs& a, cudaStream_t s);

// ---------------------------------------------------------------- decode
// Cache of one layer: [B][max_len][dkv] bf16 for K and for V.
struct KvArgs {
  int B, dkv, max_len, t_pad;
  const int* cu_seqlens;
  const int* pos;
  const __nv_bfloat16* k;   // [t_cap, dkv]
  const __nv_bfloat16* vt;  // [dkv, t_pad]
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
};
void launch_kv_store(const KvArgs& a, int t_cap, cudaStream_t s);
void launch_decode_prep(int B, int D, int V, const int* tokens, const int* cache_len, int max_len,
                        const __nv_bfloat16* embed, __nv_bfloat16* X, int* cu_seqlens, int* pos, uint32_t* status,
                        cudaStream_t s);
struct DecAttnArgs {
  int B, A, Akv, dh, dkv, G, L, P, l, max_len, t_pad, ldq, ldo;
  float scale;
  const int* cache_len;
  const uint8_t* layer_gate;
  const uint8_t* group_gate;
  const __nv_bfloat16* q;   // [B, A*dh]
  const __nv_bfloat16* k;   // [B, dkv] the new tokens' keys
  const __nv_bfloat16* vt;  // [dkv, t_pad] their values, transposed
  __nv_bfloat16* k_cache;   // this layer's [B][max_len][dkv]
  __nv_bfloat16* v_cache;
  __nv_bfloat16* out;       // [B, A*dh]
};
void launch_decode_attn(const DecAttnArgs& a, cudaStream_t s);
void launch_decode_finish(int B, int V, const float* logits, int* next_token, int* cache_len, int max_len,
                          cudaStream_t s);

// ---------------------------------------------------------------- decoder
struct ScheduleArgs {
  int B, L, G, P;
  int num_sms;              // CTAs of the persistent GEMM (one wave of tiles)
  int nsparse_rows;         // rows per tile of the QKV and gate/up lists (128, or 256 for CTA pairs)
  int nsparse_wave;         // tiles of those lists that run at once (CTAs, or CTA pairs)
  int mband;                // m-tiles per raster band of those lists (see kMBandBytes)
  int A, Akv, dh, D, Di;
  const int* cu_seqlens;
  const uint8_t* layer_gate;
  const uint8_t* group_gate;
  // per-layer outputs (layer l at offset l * cap)
  uint8_t* act;             // [L, B] sample active in layer
  int4* seg;                // [L, B] row segments {r0, r1, mask, 0}
  int4* qkv_tiles; int qkv_cap; int* qkv_count;
  int4* o_tiles; int o_cap; int* o_count;
  int4* gu_tiles; int gu_cap; int* gu_count;
  int4* dn_tiles; int dn_cap; int* dn_count;
  int4* attn_items; int attn_cap; int* attn_count;
  int* attn_next;           // [L] attention unit counters, zeroed here
  int* ks_info;             // [L][2][4]: K-split tail of the O (0) and down (1) lists, see GemmParams
  int ks_units;             // most tail shares the partial buffer holds
  uint32_t* status;
};
void launch_schedule(const ScheduleArgs& a, cudaStream_t s);

// Number of K shares the last wave of a residual GEMM's `count` tiles is cut
// into (1: no split). The persistent grid has num_sms CTAs, so the last wave
// holds r = count % num_sms tiles; it is split only when at most half full,
// into at most 8 and at most num_sms / r shares, within the `units` partial
// tiles of the workspace and the list capacity `cap`. The shares meet inside
// one launch, so the caller passes units = 0 unless every CTA of the grid is
// resident at once. Shared by the device schedule and svl_ksplit_plan.
__host__ __device__ inline int ksplit_shares(int count, int cap, int num_sms, int units) {
  if (num_sms <= 0 || count <= 0) return 1;
  const int r = count % num_sms;
  if (r == 0 || 2 * r > num_sms) return 1;
  int sp = num_sms / r;
  sp = sp < 8 ? sp : 8;
  sp = sp < units / r ? sp : units / r;
  const int room = 1 + (cap - count) / r;
  sp = sp < room ? sp : room;
  return sp < 2 ? 1 : sp;
}

// LLM-side compute controller (Sec. 3.2, Eq. 7), one block per sample: the
// budget token's state after the prefix layers plus MLP_kappa(PE(kappa)),
// the linear gate head, gates = logit > 0 for layers >= P, and (project) the
// group-only budget projection at S = S_text + k.
struct CtlArgs {
  int B, L, G, P, D, H;
  long long Dkv, Di, V;
  int project;
  const __nv_bfloat16* X;
  const int* cu_seqlens;
  const float* kappa;
  const float* budget;
  const int* k;
  const int* vis_off;
  const int* text_len;
  const __nv_bfloat16* kap_w1;
  const __nv_bfloat16* kap_w2;
  const __nv_bfloat16* gate_w;
  const float* gate_c;
  float* gate_logits;   // [B, L - P, G] or nullptr
  uint8_t* layer_gate;  // [B, L]
  uint8_t* group_gate;  // [B, L, G]
  uint32_t* flags;      // [B] or nullptr
};
void launch_controller(const CtlArgs& a, cudaStream_t s);

struct NormArgs {
  int t_cap, D, B;
  float eps;
  const __nv_bfloat16* X;
  const __nv_bfloat16* gain;
  __nv_bfloat16* Y;
  const int* cu_seqlens;
  const uint8_t* act;     // [B] or nullptr (every row)
};
void launch_rmsnorm(const NormArgs& a, cudaStream_t s);

// Fused-RMSNorm support: sums of squares of the packed rows (slot 0), norm
// gains folded into a projection's columns, and a check for unit gains.
void launch_norm_init(const __nv_bfloat16* X, const int* cu_seqlens, int B, int t_cap, int D, float* ss, int ss_ld,
                      int slots, cudaStream_t s);
cudaError_t fold_gain(const __nv_bfloat16* W, const __nv_bfloat16* g, __nv_bfloat16* out, int64_t rows, int cols,
                      cudaStream_t s);
cudaError_t gain_is_one(const __nv_bfloat16* g, int n, int* flag, cudaStream_t s);

// Final norm of each sample's last row into Y[b] (rows B..n_pad-1 zeroed).
void launch_final_last_rows(const NormArgs& a, int n_pad, cudaStream_t s);

struct AttnTcArgs {
  CUtensorMap mapQ;         // Q   [T_cap, A*dh]      boxes 64 x 128
  CUtensorMap mapVt;        // V^T [A_kv*dh, T_pad]   boxes 64 x dh
  CUtensorMap mapK64;       // K   [T_cap, A_kv*dh]   boxes 64 x 64
  CUtensorMap mapO;         // O   [T_cap, A*dh]      boxes 64 x 32 (output stores)
  const int4* items;        // {q0, q_end, r0, head}
  const int* count;
  int* next_unit;           // unit counter, zero at launch (the schedule zeroes it)
  int cap;
  int A, Akv, dh;
  float scale_log2;         // log2(e) / sqrt(dh)
  __nv_bfloat16* O;         // [T_cap, A*dh]
  int ldo;
  uint32_t* status;
};
cudaError_t launch_attention_tc(const AttnTcArgs& a, int grid, cudaStream_t s);

// One bounded wait on a barrier nobody arrives on (time-out self-test).
void launch_selftest_wait(uint32_t* status, long long cycles, cudaStream_t s);

// RoPE table: cs[i * max_seq + p] = (cos, sin)(p * theta^(-2i/dh)), double
// precision, position fastest (the lanes of a warp hold consecutive rows, so
// their reads of one frequency are contiguous).
void launch_rope_table(float2* cs, int max_seq, int dh, double theta, cudaStream_t s);

}  // namespace svl
