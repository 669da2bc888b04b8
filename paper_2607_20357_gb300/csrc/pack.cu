// Packing (Sec. 3: S = S_text + S_vis; Sec. 3.1: kept tokens form a
// compressed contiguous sequence with positions 0..S-1). Sample b occupies
// rows cu_seqlens[b]..cu_seqlens[b+1) of X: kept visual rows in ascending
// token order, then its text rows, then (with the compute controller,
// Sec. 3.2) its budget token at position S.
#include "kernels.cuh"

namespace svl {

__global__ void pack_offsets_kernel(PackArgs a) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  int t = 0;
  a.cu_seqlens[0] = 0;
  for (int b = 0; b < a.B; ++b) {
    const int kb = a.kept_off[b + 1] - a.kept_off[b];
    const int st = a.text_off[b + 1] - a.text_off[b];
    t += max(kb, 0) + max(st, 0) + (a.tok_rows ? 1 : 0);
    if (t > a.t_cap) {
      report(a.status, SVL_DEV_BAD_INDEX);
      t = a.t_cap;
    }
    a.cu_seqlens[b + 1] = t;
  }
  *a.t_total = t;
}

// One warp per output row.
__global__ void pack_gather_kernel(PackArgs a) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  const int T = *a.t_total;
  if (r >= T) return;
  int lo = 0, hi = a.B;  // sample b with cu[b] <= r < cu[b+1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (a.cu_seqlens[mid] <= r) lo = mid; else hi = mid;
  }
  const int b = lo;
  const int i = r - a.cu_seqlens[b];
  const int kb = a.kept_off[b + 1] - a.kept_off[b];
  if (lane == 0) a.pos[r] = i;
  const uint4* src;
  uint4* dst;
  int width;
  bool bad = false;
  if (i < kb) {
    const int j = a.kept_off[b] + i;
    const int n_b = a.vis_off[b + 1] - a.vis_off[b];
    int tok = a.kept_idx[j];
    if (tok < 0 || tok >= n_b) { bad = true; tok = 0; }
    src = reinterpret_cast<const uint4*>(a.vis + static_cast<size_t>(a.vis_off[b] + tok) * a.c_vis);
    width = a.c_vis;
    if (a.use_projector) {
      dst = reinterpret_cast<uint4*>(a.stage + static_cast<size_t>(j) * a.c_vis);
      if (lane == 0) a.row_map[j] = r;
    } else {
      dst = reinterpret_cast<uint4*>(a.X + static_cast<size_t>(r) * a.D);
    }
  } else if (a.tok_rows && i == kb + (a.text_off[b + 1] - a.text_off[b])) {
    src = reinterpret_cast<const uint4*>(a.tok_rows + static_cast<size_t>(b) * a.D);  // budget token
    dst = reinterpret_cast<uint4*>(a.X + static_cast<size_t>(r) * a.D);
    width = a.D;
  } else {
    int id = a.text_ids[a.text_off[b] + (i - kb)];
    if (id < 0 || id >= a.V) { bad = true; id = 0; }
    src = reinterpret_cast<const uint4*>(a.embed + static_cast<size_t>(id) * a.D);
    dst = reinterpret_cast<uint4*>(a.X + static_cast<size_t>(r) * a.D);
    width = a.D;
  }
  if (bad && lane == 0) report(a.status, SVL_DEV_BAD_INDEX);
  for (int c = lane; c < width / 8; c += 32) dst[c] = bad ? make_uint4(0, 0, 0, 0) : src[c];
}

__global__ void offsets_diff_kernel(const int* off, int* len, int B) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) len[b] = off[b + 1] - off[b];
}

void launch_offsets_diff(const int* off, int* len, int B, cudaStream_t s) {
  launch_pdl(offsets_diff_kernel, (B + 255) / 256, 256, 0, s, off, len, B);
}

void launch_pack_offsets(const PackArgs& a, cudaStream_t s) { launch_pdl(pack_offsets_kernel, 1, 32, 0, s, a); }

// One block per sample: PE(b) and the hidden layer in double, then D outputs.
__global__ void llm_budget_embed_kernel(const float* __restrict__ budget, const __nv_bfloat16* __restrict__ w1,
                                        const __nv_bfloat16* __restrict__ w2, int H, int D,
                                        __nv_bfloat16* __restrict__ out) {
  __shared__ double pe[256];
  __shared__ double hid[256];
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, i = threadIdx.x;
  const double bv = static_cast<double>(budget[b]);
  if (i < H) {
    const int half = H / 2;
    const int f = i < half ? i : i - half;
    const double arg = 1000.0 * bv * pow(10000.0, -2.0 * f / H);
    pe[i] = i < half ? sin(arg) : cos(arg);
  }
  __syncthreads();
  if (i < H) {
    double s = 0.0;
    for (int j = 0; j < H; ++j) s += static_cast<double>(__bfloat162float(w1[i * H + j])) * pe[j];
    hid[i] = s / (1.0 + exp(-s));
  }
  __syncthreads();
  for (int d = i; d < D; d += blockDim.x) {
    double s = 0.0;
    for (int j = 0; j < H; ++j) s += static_cast<double>(__bfloat162float(w2[static_cast<size_t>(d) * H + j])) * hid[j];
    out[static_cast<size_t>(b) * D + d] = __float2bfloat16_rn(static_cast<float>(s));
  }
}

void launch_llm_budget_embed(const float* budget, const __nv_bfloat16* w1, const __nv_bfloat16* w2, int H, int D,
                             int B, __nv_bfloat16* out, cudaStream_t s) {
  launch_pdl(llm_budget_embed_kernel, B, 256, 0, s, budget, w1, w2, H, D, out);
}

void launch_pack_gather(const PackArgs& a, cudaStream_t s) {
  const int rows_per_block = 8;
  const int grid = (a.t_cap + rows_per_block - 1) / rows_per_block;
  if (grid > 0) launch_pdl(pack_gather_kernel, grid, rows_per_block * 32, 0, s, a);
}

}  // namespace svl
