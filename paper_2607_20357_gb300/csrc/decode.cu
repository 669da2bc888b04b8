// Gated decode with a KV cache: one new token per sample and step, under the
// sample's prefill gates (Sec. 3.2: a gated-off head group has no keys or
// values to cache and nothing to compute; a skipped layer is bypassed). The
// paper leaves decode open (Sec. 5); the projections and the MLP run on the
// same gated tcgen05 GEMMs as the prefill with one row per sample.
//
// Cache layout (caller-owned): K then V, each [L][B][max_len][A_kv * d_head]
// bf16, position p of sample b at row p. Only the columns of KV heads of
// active groups are written and read.
#include "kernels.cuh"

namespace svl {

// Prefill: rows of the packed K [t_cap, dkv] and V^T [dkv, t_pad] of one
// layer to the cache at each row's position. 32 x 32 tiles through shared
// memory so that both the V^T reads and the cache writes are coalesced.
__global__ void kv_store_kernel(KvArgs a) {
  __shared__ __nv_bfloat16 tile[32][33];
  pdl_trigger();
  pdl_wait();
  const int T = a.cu_seqlens[a.B];
  const int r0 = blockIdx.x * 32, c0 = blockIdx.y * 32;  // packed rows, kv columns
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8 threads
  // K: row-major already, copy row by row
  for (int i = ty; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + tx;
    if (r < T && c < a.dkv) {
      const int b = find_sample(a.cu_seqlens, a.B, r);
      const int p = a.pos[r];
      if (p >= 0 && p < a.max_len)
        a.k_cache[(static_cast<size_t>(b) * a.max_len + p) * a.dkv + c] = a.k[static_cast<size_t>(r) * a.dkv + c];
    }
  }
  // V: read 32 columns of V^T (rows c) x 32 keys, write transposed
  for (int i = ty; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + tx;
    tile[i][tx] = (c < a.dkv && r < T) ? a.vt[static_cast<size_t>(c) * a.t_pad + r] : __float2bfloat16(0.f);
  }
  __syncthreads();
  for (int i = ty; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + tx;
    if (r < T && c < a.dkv) {
      const int b = find_sample(a.cu_seqlens, a.B, r);
      const int p = a.pos[r];
      if (p >= 0 && p < a.max_len) a.v_cache[(static_cast<size_t>(b) * a.max_len + p) * a.dkv + c] = tile[tx][i];
    }
  }
}

void launch_kv_store(const KvArgs& a, int t_cap, cudaStream_t s) {
  const dim3 grid((t_cap + 31) / 32, (a.dkv + 31) / 32);
  if (grid.x > 0) launch_pdl(kv_store_kernel, grid, 256, 0, s, a);
}

// Decode inputs: one row per sample (cu_seqlens = 0..B), its position is the
// cache length, its row of X the embedding of the fed token.
__global__ void decode_prep_kernel(int B, int D, int V, const int* tokens, const int* cache_len, int max_len,
                                   const __nv_bfloat16* embed, __nv_bfloat16* X, int* cu_seqlens, int* pos,
                                   uint32_t* status) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + warp;
  if (blockIdx.x == 0 && threadIdx.x == 0) cu_seqlens[0] = 0;
  if (b >= B) return;
  int id = tokens[b];
  const int len = cache_len[b];
  if (lane == 0) {
    cu_seqlens[b + 1] = b + 1;
    pos[b] = len;
    if (id < 0 || id >= V || len < 0 || len >= max_len) report(status, SVL_DEV_BAD_INDEX);
  }
  const bool bad = id < 0 || id >= V;
  if (bad) id = 0;
  const uint4* src = reinterpret_cast<const uint4*>(embed + static_cast<size_t>(id) * D);
  uint4* dst = reinterpret_cast<uint4*>(X + static_cast<size_t>(b) * D);
  for (int c = lane; c < D / 8; c += 32) dst[c] = bad ? make_uint4(0, 0, 0, 0) : src[c];
}

void launch_decode_prep(int B, int D, int V, const int* tokens, const int* cache_len, int max_len,
                        const __nv_bfloat16* embed, __nv_bfloat16* X, int* cu_seqlens, int* pos, uint32_t* status,
                        cudaStream_t s) {
  launch_pdl(decode_prep_kernel, (B + 7) / 8, 256, 0, s, B, D, V, tokens, cache_len, max_len, embed, X, cu_seqlens,
             pos, status);
}

// One block per (sample, query head) of an active group: the new token's
// query against the cached keys 0..len-1 and its own key (position len),
// softmax in float32, output row of O. The block of the first query head of
// each KV head also appends the new key and value to the cache. Each warp
// takes runs of kDecRun consecutive positions (every kDecWarps-th run),
// loading all their K and V rows before using any (lane i holds d_head / 32
// consecutive dimensions, one 4- or 8-byte load per row), and folds the run
// into its online softmax at once; the warps are merged at the end. Four
// blocks fit per SM, so a batch of 16 samples x 32 heads runs in one wave.
// Memory-bound on the cache (2 * (len + 1) * d_head * 2 bytes per head).
constexpr int kDecWarps = 8;
constexpr int kDecRun = 4;

template <int PER>  // d_head / 32: 2 or 4
SVL_DEVINL void load_row(const __nv_bfloat16* src, float* out) {
  if constexpr (PER == 4) {
    const uint2 u = *reinterpret_cast<const uint2*>(src);
    const float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
    out[0] = a.x; out[1] = a.y; out[2] = b.x; out[3] = b.y;
  } else {
    const float2 a = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(src));
    out[0] = a.x; out[1] = a.y;
  }
}

template <int PER>
__global__ void __launch_bounds__(kDecWarps * 32, 4) decode_attn_kernel(DecAttnArgs a) {
  __shared__ float sm_m[kDecWarps], sm_l[kDecWarps];
  __shared__ float sm_o[kDecWarps][128];
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, h = blockIdx.y;
  const int G = a.G, hpg = a.A / G, g = h / hpg;
  if (!(a.layer_gate[b * a.L + a.l] && a.group_gate[(static_cast<size_t>(b) * a.L + a.l) * G + g]) && a.l >= a.P)
    return;  // gated off: no keys, no values, no output
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int dh = a.dh, kvh = h / (a.A / a.Akv);
  const int len = a.cache_len[b];
  if (len < 0 || len >= a.max_len) return;  // reported by decode_prep
  const size_t cbase = static_cast<size_t>(b) * a.max_len * a.dkv + static_cast<size_t>(kvh) * dh + lane * PER;
  float q[PER], kn[PER], vn[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int d = lane * PER + i;
    q[i] = __bfloat162float(a.q[static_cast<size_t>(b) * a.ldq + h * dh + d]) * a.scale;
    kn[i] = __bfloat162float(a.k[static_cast<size_t>(b) * a.dkv + kvh * dh + d]);
    vn[i] = __bfloat162float(a.vt[static_cast<size_t>(kvh * dh + d) * a.t_pad + b]);
  }
  if (h % (a.A / a.Akv) == 0 && warp == 0) {
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      a.k_cache[cbase + static_cast<size_t>(len) * a.dkv + i] = __float2bfloat16_rn(kn[i]);
      a.v_cache[cbase + static_cast<size_t>(len) * a.dkv + i] = __float2bfloat16_rn(vn[i]);
    }
  }
  float m = -INFINITY, l = 0.f, o[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) o[i] = 0.f;
  for (int p0 = warp * kDecRun; p0 <= len; p0 += kDecWarps * kDecRun) {
    float kk[kDecRun][PER], vv[kDecRun][PER], sc[kDecRun];
#pragma unroll
    for (int u = 0; u < kDecRun; ++u) {
      const int p = p0 + u;
      if (p < len) {
        load_row<PER>(a.k_cache + cbase + static_cast<size_t>(p) * a.dkv, kk[u]);
        load_row<PER>(a.v_cache + cbase + static_cast<size_t>(p) * a.dkv, vv[u]);
      } else {
#pragma unroll
        for (int i = 0; i < PER; ++i) {
          kk[u][i] = p == len ? kn[i] : 0.f;
          vv[u][i] = p == len ? vn[i] : 0.f;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kDecRun; ++u) {
      float d = 0.f;
#pragma unroll
      for (int i = 0; i < PER; ++i) d = fmaf(q[i], kk[u][i], d);
      sc[u] = d;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
#pragma unroll
      for (int u = 0; u < kDecRun; ++u) sc[u] += __shfl_xor_sync(0xffffffffu, sc[u], off);
    float mr = m;
#pragma unroll
    for (int u = 0; u < kDecRun; ++u)
      if (p0 + u <= len) mr = fmaxf(mr, sc[u]);
    const float corr = __expf(m - mr);
    l *= corr;
#pragma unroll
    for (int i = 0; i < PER; ++i) o[i] *= corr;
#pragma unroll
    for (int u = 0; u < kDecRun; ++u) {
      const float e = p0 + u <= len ? __expf(sc[u] - mr) : 0.f;
      l += e;
#pragma unroll
      for (int i = 0; i < PER; ++i) o[i] = fmaf(e, vv[u][i], o[i]);
    }
    m = mr;
  }
  if (lane == 0) {
    sm_m[warp] = m;
    sm_l[warp] = l;
  }
#pragma unroll
  for (int i = 0; i < PER; ++i) sm_o[warp][lane * PER + i] = o[i];
  __syncthreads();
  if (warp == 0) {
    float M = -INFINITY;
    for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, sm_m[w]);
    float L = 0.f, acc[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = 0.f;
    for (int w = 0; w < kDecWarps; ++w) {
      const float f = sm_m[w] == -INFINITY ? 0.f : __expf(sm_m[w] - M);
      L += sm_l[w] * f;
#pragma unroll
      for (int i = 0; i < PER; ++i) acc[i] += sm_o[w][lane * PER + i] * f;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i)
      a.out[static_cast<size_t>(b) * a.ldo + h * dh + lane * PER + i] = __float2bfloat16_rn(acc[i] * inv);
  }
}

void launch_decode_attn(const DecAttnArgs& a, cudaStream_t s) {
  if (a.dh == 128)
    launch_pdl(decode_attn_kernel<4>, dim3(a.B, a.A), kDecWarps * 32, 0, s, a);
  else
    launch_pdl(decode_attn_kernel<2>, dim3(a.B, a.A), kDecWarps * 32, 0, s, a);
}

// Greedy next token per sample (largest logit; equal logits: lower id) and
// the cache length advanced by the fed token. One 1024-thread block per
// sample; with V a multiple of 4 each thread reads float4s (4 consecutive ids,
// kept in id order, so the tie rule holds).
constexpr int kFinThreads = 1024;

SVL_DEVINL void arg_better(float x, int v, float& best, int& idx) {
  if (x > best || (x == best && v < idx)) {
    best = x;
    idx = v;
  }
}

__global__ void __launch_bounds__(kFinThreads) decode_finish_kernel(int B, int V, const float* logits, int* next_token,
                                                                    int* cache_len) {
  __shared__ float bv[kFinThreads / 32];
  __shared__ int bi[kFinThreads / 32];
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* row = logits + static_cast<size_t>(b) * V;
  float best = -INFINITY;
  int idx = 0x7fffffff;
  if ((V & 3) == 0) {
    const float4* r4 = reinterpret_cast<const float4*>(row);
    for (int c = tid; c < V / 4; c += kFinThreads) {
      const float4 x = r4[c];
      arg_better(x.x, 4 * c, best, idx);
      arg_better(x.y, 4 * c + 1, best, idx);
      arg_better(x.z, 4 * c + 2, best, idx);
      arg_better(x.w, 4 * c + 3, best, idx);
    }
  } else {
    for (int v = tid; v < V; v += kFinThreads) arg_better(row[v], v, best, idx);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, off);
    const int oi = __shfl_xor_sync(0xffffffffu, idx, off);
    arg_better(ob, oi, best, idx);
  }
  if (lane == 0) {
    bv[warp] = best;
    bi[warp] = idx;
  }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < kFinThreads / 32; ++w) arg_better(bv[w], bi[w], best, idx);
    if (next_token) next_token[b] = idx == 0x7fffffff ? 0 : idx;
    cache_len[b] += 1;
  }
}

void launch_decode_finish(int B, int V, const float* logits, int* next_token, int* cache_len, cudaStream_t s) {
  launch_pdl(decode_finish_kernel, B, kFinThreads, 0, s, B, V, logits, next_token, cache_len);
}

}  // namespace svl
