// Token controller (Sec. 3.1; Sec. 3.3 "Inference"): budget embedding,
// budget -> k from Eq. 8, per-sample top-k by radix select, stable compaction.
// The token scores themselves come from the tcgen05 GEMM (EPI_SCORE).
#include "kernels.cuh"

namespace svl {

// e_b = W_b2 SiLU(W_b1 PE(b)), PE(b) = [sin(1000 b w_i) | cos(1000 b w_i)],
// w_i = 10000^(-2i/H) (Eq. 5). One block per sample. The argument reaches
// 1000 rad, so it is formed and reduced to [-pi, pi] in double precision
// before the single-precision sine and cosine (error about 1e-7 either way);
// the two H x H products run in fp32, four threads per output.
constexpr double kTwoPi = 6.283185307179586;

SVL_DEVINL void budget_matvec(const __nv_bfloat16* __restrict__ w, const float* x, int H, float* y, bool silu) {
  const int i = threadIdx.x, part = i & 3;
  for (int o0 = 0; o0 < H; o0 += blockDim.x / 4) {
    const int o = o0 + i / 4;
    float s = 0.f;
    if (o < H)
      for (int j = part; j < H; j += 4) s = fmaf(__bfloat162float(w[static_cast<size_t>(o) * H + j]), x[j], s);
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    if (o < H && part == 0) y[o] = silu ? s / (1.f + expf(-s)) : s;
  }
}

__global__ void budget_embed_kernel(const float* __restrict__ budget, const __nv_bfloat16* __restrict__ w1,
                                    const __nv_bfloat16* __restrict__ w2, int H, float* __restrict__ e_b) {
  __shared__ float pe[256];
  __shared__ float hid[256];
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, i = threadIdx.x;
  if (i < H) {
    const int half = H / 2;
    const int f = i < half ? i : i - half;
    const double omega = pow(10000.0, -2.0 * f / H);
    const double arg = 1000.0 * static_cast<double>(budget[b]) * omega;
    const float r = static_cast<float>(arg - rint(arg / kTwoPi) * kTwoPi);
    pe[i] = i < half ? sinf(r) : cosf(r);
  }
  __syncthreads();
  budget_matvec(w1, pe, H, hid, true);
  __syncthreads();
  budget_matvec(w2, hid, H, e_b + static_cast<size_t>(b) * H, false);
}

// Orderable key: unsigned comparison of keys matches float comparison.
SVL_DEVINL uint32_t order_key(float z) {
  if (z == 0.0f) z = 0.0f;  // -0 and +0 are equal logits
  const uint32_t u = __float_as_uint(z);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive block-wide prefix sum of one int per thread (blockDim.x <= 1024).
SVL_DEVINL int block_exclusive_scan(int v, int* total, int* warp_sums) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nw) warp_sums[lane] = w;  // inclusive
  }
  __syncthreads();
  const int base = warp > 0 ? warp_sums[warp - 1] : 0;
  *total = warp_sums[nw - 1];
  __syncthreads();
  return base + x - v;
}

// One block per sample: k from the budget (largest k with Eq. 8 cost within
// b * C_full), then the k largest logits (ties: lower index), written in
// ascending index order to kept_local[vis_off[b] ...].
//
// Under the paper's own rule (a.gate_logits set; Sec. 3.1 and Sec. 3.3
// "Inference") the gates are the compute controller's logits > 0 (prefix
// layers always on), k is capped by the number of logits z > 0 (sigma > 0.5),
// and when no visual token fits the budget, the fewest active groups of layers
// l >= P that make it fit are switched off, lowest logit first (equal logits:
// lower (l, j) first); the projected gates are written out.
__global__ void __launch_bounds__(kSelectThreads) select_kernel(SelectArgs a) {
  __shared__ int hist[256];
  __shared__ int warp_sums[32];
  __shared__ int best_k;
  __shared__ int s_prefix_cnt[2];
  __shared__ long long n_on_sum;  // updated with 64-bit atomics
  __shared__ int n_pos, keep_groups;
  __shared__ double kappa_sum;
  pdl_trigger();
  pdl_wait();

  const int b = blockIdx.x, tid = threadIdx.x;
  const int v0 = a.vis_off[b], v1 = a.vis_off[b + 1];
  const int n = max(0, v1 - v0);
  const long long s_text = a.text_len[b];

  // ---- k from the budget (Eq. 8, exact integers scaled by G)
  if (tid == 0) {
    n_on_sum = 0;
    best_k = -1;
    n_pos = 0;
    keep_groups = -1;
    kappa_sum = 0.0;
  }
  __syncthreads();
  const float* gl = a.gate_logits ? a.gate_logits + static_cast<size_t>(b) * a.L * a.G : nullptr;
  auto active = [&](int idx) -> bool {
    const int l = idx / a.G;
    if (l < a.P) return true;
    return gl ? gl[idx] > 0.f : (a.layer_gate[b * a.L + l] && a.group_gate[b * a.L * a.G + idx]);
  };
  {
    // active (layer, group) pairs of this sample; not needed (and no gates
    // given) when the gates are decided later
    int on = 0;
    if (!a.threshold_only)
      for (int idx = tid; idx < a.L * a.G; idx += blockDim.x) on += active(idx) ? 1 : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) on += __shfl_xor_sync(0xffffffffu, on, o);
    if ((tid & 31) == 0 && on) atomicAdd(reinterpret_cast<unsigned long long*>(&n_on_sum), static_cast<unsigned long long>(on));
    if (gl || a.threshold_only) {
      int pos = 0;  // logits z > 0, i.e. sigma(z) > 0.5
      for (int i = tid; i < n; i += blockDim.x) pos += a.scores[v0 + i] > 0.f ? 1 : 0;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) pos += __shfl_xor_sync(0xffffffffu, pos, o);
      if ((tid & 31) == 0 && pos) atomicAdd(&n_pos, pos);
    }
    if (a.kappa) {
      // survival rate kappa = sum sigma(z_i) / N that conditions the compute controller (Sec. 3.2)
      double sg = 0.0;
      for (int i = tid; i < n; i += blockDim.x) sg += 1.0 / (1.0 + exp(-static_cast<double>(a.scores[v0 + i])));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sg += __shfl_xor_sync(0xffffffffu, sg, o);
      if ((tid & 31) == 0) atomicAdd(&kappa_sum, sg);
    }
  }
  __syncthreads();
  int k;
  uint32_t flags = 0;
  const int kc = a.keep_count ? a.keep_count[b] : -1;
  if (tid == 0 && a.kappa) a.kappa[b] = n > 0 ? static_cast<float>(kappa_sum / n) : 0.f;
  if (kc >= 0) {
    k = min(kc, n);
  } else if (a.threshold_only) {
    k = n_pos;  // the compute controller decides the gates later
  } else {
    const long long D = a.D, Dkv = a.Dkv, Di = a.Di, V = a.V, G = a.G, L = a.L;
    const long long lin = 4 * D * D + 4 * D * Dkv + 6 * D * Di;
    const long long S_full = n + s_text;
    const long long c_full = G * L * (lin * S_full + 4 * D * S_full * S_full) + G * 2 * D * V * S_full;
    const double limit = static_cast<double>(a.budget[b]) * static_cast<double>(c_full);
    long long mine = -1;
    for (int kk = tid; kk <= n; kk += blockDim.x) {
      const long long S = s_text + kk;
      const long long cost = n_on_sum * (lin * S + 4 * D * S * S) + G * 2 * D * V * S;
      if (static_cast<double>(cost) <= limit) mine = max(mine, static_cast<long long>(kk));
    }
    // cost grows with k, so the feasible set is a prefix: take the max
    if (mine >= 0) atomicMax(&best_k, static_cast<int>(mine));
    __syncthreads();
    if (best_k >= 0) {
      k = gl ? min(best_k, n_pos) : best_k;
    } else if (!gl) {
      k = 0;
      flags |= SVL_FLAG_OVER_BUDGET;
    } else {
      // paper rule: no visual token fits, so head groups go. The most groups
      // that still fit with the text alone (prefix groups cannot go):
      k = 0;
      const long long n_min = static_cast<long long>(min(a.P, a.L)) * G;
      const long long per = lin * s_text + 4 * D * s_text * s_text, lm = G * 2 * D * V * s_text;
      for (long long nk = n_min + tid; nk < n_on_sum; nk += blockDim.x)
        if (static_cast<double>(nk * per + lm) <= limit) atomicMax(&keep_groups, static_cast<int>(nk));
      __syncthreads();
      if (n_on_sum > n_min) flags |= SVL_FLAG_GROUPS_DROPPED;
      const bool over = keep_groups < 0;  // even the prefix layers alone exceed the budget
      if (over) flags |= SVL_FLAG_OVER_BUDGET;
      __syncthreads();
      if (over && tid == 0) keep_groups = static_cast<int>(n_min);
    }
  }
  if (gl) {
    // projected gates: the (n_on - keep_groups) lowest-logit active groups
    // of layers >= P are off (none unless the fallback ran)
    __syncthreads();
    const int drop = keep_groups < 0 ? 0 : static_cast<int>(n_on_sum) - keep_groups;
    uint8_t* go = a.group_gate_out + static_cast<size_t>(b) * a.L * a.G;
    for (int idx = tid; idx < a.L * a.G; idx += blockDim.x) {
      bool on = active(idx);
      if (on && drop > 0 && idx >= a.P * a.G) {
        const float v = gl[idx];
        int rank = 0;
        for (int j = a.P * a.G; j < a.L * a.G; ++j)
          if (active(j) && (gl[j] < v || (gl[j] == v && j < idx))) ++rank;
        on = rank >= drop;
      }
      go[idx] = on ? 1 : 0;
    }
    __syncthreads();
    for (int l = tid; l < a.L; l += blockDim.x) {
      int any = 0;
      for (int j = 0; j < a.G; ++j) any |= go[l * a.G + j];
      a.layer_gate_out[static_cast<size_t>(b) * a.L + l] = any ? 1 : 0;
    }
  }
  if (tid == 0) {
    a.k_out[b] = k;
    if (a.flags) a.flags[b] = flags;
  }

  const float* z = a.scores + v0;
  int* out = a.kept_local + v0;
  if (k == 0) return;
  if (k >= n) {
    for (int i = tid; i < n; i += blockDim.x) out[i] = i;
    return;
  }

  // ---- radix select of the k-th largest key, 8 bits per pass, MSB first
  uint32_t prefix = 0, mask = 0;
  int remaining = k;  // keys still to take among those matching `prefix`
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < n; i += blockDim.x) {
      const uint32_t key = order_key(z[i]);
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 0xFF], 1);
    }
    __syncthreads();
    if (tid < 32) {
      // warp 0: counts above each digit (suffix sums from 255 down), then the
      // largest digit d whose keys with digit >= d reach `remaining`
      int cnt[8], sum = 0;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        cnt[u] = hist[255 - (tid * 8 + u)];  // lane t holds digits 255-8t .. 248-8t
        sum += cnt[u];
      }
      int incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += y;
      }
      int above = incl - sum;  // keys with a digit above this lane's first digit
      int found = -1, found_above = 0;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (found < 0 && above + cnt[u] >= remaining) {
          found = 255 - (tid * 8 + u);
          found_above = above;
        }
        above += cnt[u];
      }
      const unsigned ballot = __ballot_sync(0xffffffffu, found >= 0);
      const int first = ballot ? __ffs(ballot) - 1 : 31;
      const int d = __shfl_sync(0xffffffffu, found, first);
      const int ab = __shfl_sync(0xffffffffu, found_above, first);
      if (tid == 0) {
        s_prefix_cnt[0] = d < 0 ? 0 : d;
        s_prefix_cnt[1] = remaining - (d < 0 ? 0 : ab);
      }
    }
    __syncthreads();
    prefix |= static_cast<uint32_t>(s_prefix_cnt[0]) << shift;
    mask |= 0xFFu << shift;
    remaining = s_prefix_cnt[1];
    __syncthreads();
  }
  const uint32_t tau = prefix;  // key of the k-th largest logit
  // keys > tau are kept; of the keys == tau, the `remaining` lowest indices

  // ---- ordered pass: ranks of equal keys and output positions by index
  int eq_before = 0, kept_before = 0;
  for (int base = 0; base < n; base += blockDim.x) {
    const int i = base + tid;
    uint32_t key = 0;
    if (i < n) key = order_key(z[i]);
    const int is_eq = (i < n && key == tau) ? 1 : 0;
    int eq_total;
    const int eq_rank = eq_before + block_exclusive_scan(is_eq, &eq_total, warp_sums);
    const int keep = (i < n && (key > tau || (is_eq && eq_rank < remaining))) ? 1 : 0;
    int keep_total;
    const int pos = kept_before + block_exclusive_scan(keep, &keep_total, warp_sums);
    if (keep) out[pos] = i;
    eq_before += eq_total;
    kept_before += keep_total;
  }
}

// Compacts the per-sample kept lists: kept_off[b] = k_0 + ... + k_{b-1}.
__global__ void compact_kernel(int B, const int* __restrict__ vis_off, const int* __restrict__ k,
                               const int* __restrict__ kept_local, int* __restrict__ kept_idx,
                               int* __restrict__ kept_off, int* __restrict__ kept_total) {
  __shared__ int off;
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  if (threadIdx.x == 0) off = 0;
  __syncthreads();
  int part = 0;  // k of the samples before b, summed by all threads
  for (int i = threadIdx.x; i < b; i += blockDim.x) part += k[i];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
  if ((threadIdx.x & 31) == 0 && part) atomicAdd(&off, part);
  __syncthreads();
  if (threadIdx.x == 0) {
    kept_off[b] = off;
    if (b == B - 1) {
      kept_off[B] = off + k[b];
      if (kept_total) *kept_total = off + k[b];
    }
  }
  const int kb = k[b];
  const int* src = kept_local + vis_off[b];
  for (int i = threadIdx.x; i < kb; i += blockDim.x) kept_idx[off + i] = src[i];
}

void launch_budget_embed(const float* budget, const __nv_bfloat16* w1, const __nv_bfloat16* w2, int H, int B,
                         float* e_b, cudaStream_t s) {
  launch_pdl(budget_embed_kernel, B, 256, 0, s, budget, w1, w2, H, e_b);
}

void launch_select(const SelectArgs& a, int B, cudaStream_t s) {
  launch_pdl(select_kernel, B, kSelectThreads, 0, s, a);
}

void launch_compact(int B, const int* vis_off, const int* k, const int* kept_local, int* kept_idx, int* kept_off,
                    int* kept_total, cudaStream_t s) {
  launch_pdl(compact_kernel, B, 256, 0, s, B, vis_off, k, kept_local, kept_idx, kept_off, kept_total);
}

}  // namespace svl
