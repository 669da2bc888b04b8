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
// each KV head also appends the new key and value to the cache. Each of the
// 8 warps takes a contiguous run of positions, 32 at a time: lane j scores
// key j on its own (its whole K row as 16-byte loads against q in shared
// memory, no shuffles per key), the warp folds the 32 scores into its online
// softmax, then every lane accumulates its d_head / 32 output dimensions over
// the 32 V rows (independent loads). The warps are merged at the end.
// Memory-bound on the cache (2 * (len + 1) * d_head * 2 bytes per head).
constexpr int kDecWarps = 8;

template <int DH>  // d_head: 64 or 128
__global__ void __launch_bounds__(kDecWarps * 32, 4) decode_attn_kernel(DecAttnArgs a) {
  constexpr int PER = DH / 32;
  __shared__ __align__(16) float sq[DH];  // q * scale
  __shared__ __align__(16) float snv[DH];  // the new value row
  __shared__ float sm_m[kDecWarps], sm_l[kDecWarps];
  __shared__ float sm_o[kDecWarps][DH];
  __shared__ float sp[kDecWarps][32];
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, h = blockIdx.y;
  const int G = a.G, hpg = a.A / G, g = h / hpg;
  if (!(a.layer_gate[b * a.L + a.l] && a.group_gate[(static_cast<size_t>(b) * a.L + a.l) * G + g]) && a.l >= a.P)
    return;  // gated off: no keys, no values, no output
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  const int kvh = h / (a.A / a.Akv);
  const int len = a.cache_len[b];
  if (len < 0 || len >= a.max_len) {
    // full (or corrupt) cache, reported by decode_prep: the head's output is
    // zero, so the step's logits for this sample are defined, and nothing is
    // appended
    if (tid < DH) a.out[static_cast<size_t>(b) * a.ldo + h * DH + tid] = __float2bfloat16(0.f);
    return;
  }
  const __nv_bfloat16* knew = a.k + static_cast<size_t>(b) * a.dkv + kvh * DH;
  if (tid < DH) {
    sq[tid] = __bfloat162float(a.q[static_cast<size_t>(b) * a.ldq + h * DH + tid]) * a.scale;
    const __nv_bfloat16 vnew = a.vt[static_cast<size_t>(kvh * DH + tid) * a.t_pad + b];
    snv[tid] = __bfloat162float(vnew);
    if (h % (a.A / a.Akv) == 0) {  // append the new key and value to the cache
      const size_t at = (static_cast<size_t>(b) * a.max_len + len) * a.dkv + kvh * DH + tid;
      a.k_cache[at] = knew[tid];
      a.v_cache[at] = vnew;
    }
  }
  __syncthreads();
  const size_t cbase = static_cast<size_t>(b) * a.max_len * a.dkv + static_cast<size_t>(kvh) * DH;
  const int n = len + 1, per_warp = (n + kDecWarps - 1) / kDecWarps;
  const int p_begin = warp * per_warp, p_end = min(n, p_begin + per_warp);
  float m = -INFINITY, l = 0.f, o[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) o[i] = 0.f;
  for (int p0 = p_begin; p0 < p_end; p0 += 32) {
    const int p = p0 + lane;
    float sc = -INFINITY;
    if (p < p_end) {
      const uint4* kr = reinterpret_cast<const uint4*>(p < len ? a.k_cache + cbase + static_cast<size_t>(p) * a.dkv
                                                               : knew);
      uint4 u[DH / 8];
#pragma unroll
      for (int c = 0; c < DH / 8; ++c) u[c] = kr[c];
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < DH / 8; ++c) {
        const float4 q0 = *reinterpret_cast<const float4*>(sq + 8 * c);
        const float4 q1 = *reinterpret_cast<const float4*>(sq + 8 * c + 4);
        const float2 k0 = unpack_bf16x2(u[c].x), k1 = unpack_bf16x2(u[c].y), k2 = unpack_bf16x2(u[c].z),
                     k3 = unpack_bf16x2(u[c].w);
        acc = fmaf(q0.x, k0.x, acc);
        acc = fmaf(q0.y, k0.y, acc);
        acc = fmaf(q0.z, k1.x, acc);
        acc = fmaf(q0.w, k1.y, acc);
        acc = fmaf(q1.x, k2.x, acc);
        acc = fmaf(q1.y, k2.y, acc);
        acc = fmaf(q1.z, k3.x, acc);
        acc = fmaf(q1.w, k3.y, acc);
      }
      sc = acc;
    }
    float mx = sc;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    const float mn = fmaxf(m, mx);
    const float e = p < p_end ? __expf(sc - mn) : 0.f;
    float es = e;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) es += __shfl_xor_sync(0xffffffffu, es, off);
    const float corr = __expf(m - mn);  // 0 while m is -inf
    l = l * corr + es;
#pragma unroll
    for (int i = 0; i < PER; ++i) o[i] *= corr;
    m = mn;
    sp[warp][lane] = e;
    __syncwarp();
    const int nk = min(32, p_end - p0);
#pragma unroll 8
    for (int j = 0; j < nk; ++j) {
      const int pj = p0 + j;
      const float ej = sp[warp][j];
      float vv[PER];
      if (pj < len) {
        const __nv_bfloat16* vr = a.v_cache + cbase + static_cast<size_t>(pj) * a.dkv + lane * PER;
        if constexpr (PER == 4) {
          const uint2 w = *reinterpret_cast<const uint2*>(vr);
          const float2 v0 = unpack_bf16x2(w.x), v1 = unpack_bf16x2(w.y);
          vv[0] = v0.x; vv[1] = v0.y; vv[2] = v1.x; vv[3] = v1.y;
        } else {
          const float2 v0 = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(vr));
          vv[0] = v0.x; vv[1] = v0.y;
        }
      } else {
#pragma unroll
        for (int i = 0; i < PER; ++i) vv[i] = snv[lane * PER + i];
      }
#pragma unroll
      for (int i = 0; i < PER; ++i) o[i] = fmaf(ej, vv[i], o[i]);
    }
    __syncwarp();
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
      a.out[static_cast<size_t>(b) * a.ldo + h * DH + lane * PER + i] = __float2bfloat16_rn(acc[i] * inv);
  }
}

void launch_decode_attn(const DecAttnArgs& a, cudaStream_t s) {
  if (a.dh == 128)
    launch_pdl(decode_attn_kernel<128>, dim3(a.B, a.A), kDecWarps * 32, 0, s, a);
  else
    launch_pdl(decode_attn_kernel<64>, dim3(a.B, a.A), kDecWarps * 32, 0, s, a);
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
                                                                    int* cache_len, int max_len) {
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
    // a sample whose cache was already full took no step: its length stays
    // and it has no next token
    const int len = cache_len[b];
    const bool stepped = len >= 0 && len < max_len;
    if (next_token) next_token[b] = !stepped ? -1 : (idx == 0x7fffffff ? 0 : idx);
    if (stepped) cache_len[b] = len + 1;
  }
}

void launch_decode_finish(int B, int V, const float* logits, int* next_token, int* cache_len, int max_len,
                          cudaStream_t s) {
  launch_pdl(decode_finish_kernel, B, kFinThreads, 0, s, B, V, logits, next_token, cache_len, max_len);
}

}  // namespace svl
