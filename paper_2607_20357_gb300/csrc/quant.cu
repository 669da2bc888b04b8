// e4m3 operands of the gated projections (FP8 weights, which the paper
// calls orthogonal to its method, Sec. 5). Every row -- an output channel of
// a weight matrix, or an activation row feeding one of the four gated GEMMs
// -- is scaled so that its largest magnitude maps to 448, the largest finite
// e4m3 value, and rounded to nearest even with saturation:
//
//   amax = max |x|, inv = 448 / amax, scale = amax / 448 (float32, correctly
//   rounded; 0 and 0 when amax = 0), code = e4m3(x * inv).
//
// With a gain vector (the RMSNorm gain of the projection's input norm) the
// row quantised is x * gain, each product exact in float32 (two bf16
// factors). The norm's 1/rms(x) is a factor of the whole row, so the codes of
// x * gain are those of RMSNorm(x) * gain and the GEMM applies 1/rms with the
// row's scale after the product.
//
// The GEMM multiplies codes and scales its accumulator by both rows' scales.
#include <algorithm>

#include "kernels.cuh"

namespace svl {

constexpr int kQuantWarps = 8;

// Eight bf16 ones: the gain of a row quantised as it is.
SVL_DEVINL uint4 ones8() { return make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u); }

// The eight values of a 16-byte chunk times their gains, in float32 (exact:
// the product of two bf16 values has at most 16 significant bits).
SVL_DEVINL void scaled8(const uint4 x, const uint4 g, float f[8]) {
  const uint32_t xw[4] = {x.x, x.y, x.z, x.w}, gw[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 a = unpack_bf16x2(xw[q]), b = unpack_bf16x2(gw[q]);
    f[2 * q] = __fmul_rn(a.x, b.x);
    f[2 * q + 1] = __fmul_rn(a.y, b.y);
  }
}

// e4m3 codes of eight values times inv (each product rounded to float32).
SVL_DEVINL uint2 codes8(const float f[8], float inv) {
  uint2 o;
  o.x = static_cast<uint32_t>(e4m3x2(__fmul_rn(f[0], inv), __fmul_rn(f[1], inv))) |
        (static_cast<uint32_t>(e4m3x2(__fmul_rn(f[2], inv), __fmul_rn(f[3], inv))) << 16);
  o.y = static_cast<uint32_t>(e4m3x2(__fmul_rn(f[4], inv), __fmul_rn(f[5], inv))) |
        (static_cast<uint32_t>(e4m3x2(__fmul_rn(f[6], inv), __fmul_rn(f[7], inv))) << 16);
  return o;
}

// One warp per row, two passes (rows wider than 16,384 codes).
__global__ void __launch_bounds__(kQuantWarps * 32) quant_rows_kernel(QuantArgs a) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t r = static_cast<int64_t>(blockIdx.x) * kQuantWarps + warp;
  int64_t rows = a.rows;
  if (a.cu_seqlens) rows = min(rows, static_cast<int64_t>(a.cu_seqlens[a.B]));
  if (r >= rows) return;
  int mask = (1 << a.G) - 1;
  if (a.group_gate && a.l >= a.P) {
    const int b = find_sample(a.cu_seqlens, a.B, static_cast<int>(r));
    const size_t bl = static_cast<size_t>(b) * a.L + a.l;
    mask = 0;
    if (a.layer_gate[bl])
      for (int j = 0; j < a.G; ++j) mask |= a.group_gate[bl * a.G + j] ? (1 << j) : 0;
  }
  const __nv_bfloat16* src = a.src + r * a.ld_src;
  float amax = 0.f;
  for (int j = 0; j < a.G; ++j) {
    if (!((mask >> j) & 1)) continue;
    const uint4* s4 = reinterpret_cast<const uint4*>(src + static_cast<size_t>(j) * a.kg);
    const uint4* g4 = a.gain ? reinterpret_cast<const uint4*>(a.gain + static_cast<size_t>(j) * a.kg) : nullptr;
    for (int c = lane; c < a.kg / 8; c += 32) {
      float f[8];
      scaled8(s4[c], g4 ? g4[c] : ones8(), f);
#pragma unroll
      for (int q = 0; q < 8; ++q) amax = fmaxf(amax, fabsf(f[q]));
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
  const float inv = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
  uint8_t* dst = a.dst + r * a.ld_dst;
  for (int j = 0; j < a.G; ++j) {
    const bool on = (mask >> j) & 1;
    const uint4* s4 = reinterpret_cast<const uint4*>(src + static_cast<size_t>(j) * a.kg);
    const uint4* g4 = a.gain ? reinterpret_cast<const uint4*>(a.gain + static_cast<size_t>(j) * a.kg) : nullptr;
    uint2* d8 = reinterpret_cast<uint2*>(dst + static_cast<size_t>(j) * a.kgp);
    for (int c = lane; c < a.kgp / 8; c += 32) {
      uint2 o = make_uint2(0, 0);
      if (on && c < a.kg / 8) {
        float f[8];
        scaled8(s4[c], g4 ? g4[c] : ones8(), f);
        o = codes8(f, inv);
      }
      d8[c] = o;
    }
  }
  if (lane == 0) a.scale[r] = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
}

// 128-thread CTAs walking the rows (row = blockIdx.x + i * gridDim.x, so a
// grid sized for the SMs serves any row count without idle CTAs): thread t
// holds the row's 16-byte chunks t, t + 128, ... (NCH of them) in registers
// between the amax and the code pass, so each bf16 value is read once.
constexpr int kQuantThreads = 128;

template <int NCH, bool GAIN>
__global__ void __launch_bounds__(kQuantThreads) quant_row_cta_kernel(QuantArgs a) {
  __shared__ float red[2][kQuantThreads / 32];
  __shared__ int s_mask[2];
  pdl_trigger();
  pdl_wait();
  int64_t rows = a.rows;
  if (a.cu_seqlens) rows = min(rows, static_cast<int64_t>(a.cu_seqlens[a.B]));
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int par = 0;  // the shared slots alternate between consecutive rows
  for (int64_t r = blockIdx.x; r < rows; r += gridDim.x, par ^= 1) {
    if (tid == 0) {
      int mask = (1 << a.G) - 1;
      if (a.group_gate && a.l >= a.P) {
        const int b = find_sample(a.cu_seqlens, a.B, static_cast<int>(r));
        const size_t bl = static_cast<size_t>(b) * a.L + a.l;
        mask = 0;
        if (a.layer_gate[bl])
          for (int j = 0; j < a.G; ++j) mask |= a.group_gate[bl * a.G + j] ? (1 << j) : 0;
      }
      s_mask[par] = mask;
    }
    __syncthreads();
    const int mask = s_mask[par];
    const int per_g = a.kgp / 8, src_per_g = a.kg / 8, nchunk = a.G * per_g;
    const __nv_bfloat16* src = a.src + r * a.ld_src;
    uint4 v[NCH], gv[GAIN ? NCH : 1];
    float amax = 0.f;
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      const int c = tid + i * kQuantThreads;
      v[i] = make_uint4(0, 0, 0, 0);
      if (GAIN) gv[i] = ones8();
      if (c < nchunk) {
        const int j = c / per_g, cc = c - j * per_g;
        if (((mask >> j) & 1) && cc < src_per_g) {
          const size_t col = static_cast<size_t>(j) * a.kg + static_cast<size_t>(cc) * 8;
          v[i] = *reinterpret_cast<const uint4*>(src + col);
          if (GAIN) gv[i] = *reinterpret_cast<const uint4*>(a.gain + col);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      float f[8];
      scaled8(v[i], GAIN ? gv[i] : ones8(), f);
#pragma unroll
      for (int q = 0; q < 8; ++q) amax = fmaxf(amax, fabsf(f[q]));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
    if (lane == 0) red[par][warp] = amax;
    __syncthreads();
    amax = fmaxf(fmaxf(red[par][0], red[par][1]), fmaxf(red[par][2], red[par][3]));
    const float inv = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
    uint8_t* dst = a.dst + r * a.ld_dst;
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      const int c = tid + i * kQuantThreads;
      if (c < nchunk) {
        float f[8];
        scaled8(v[i], GAIN ? gv[i] : ones8(), f);
        // chunk c of the padded row sits at byte 8 c (groups are kgp apart)
        *reinterpret_cast<uint2*>(dst + static_cast<size_t>(c) * 8) = codes8(f, inv);
      }
    }
    if (tid == 0) a.scale[r] = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
  }
}

cudaError_t launch_quant_rows(const QuantArgs& a, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
  }
  const int64_t chunks = static_cast<int64_t>(a.G) * (a.kgp / 8);
  // enough CTAs to fill every SM (16 resident for the 4-chunk rows, fewer
  // for the wider ones, which are limited by registers)
  auto grid_for = [&](int per_sm) {
    return dim3(static_cast<unsigned>(std::min<int64_t>(a.rows, static_cast<int64_t>(sms) * per_sm)));
  };
  const dim3 grid = grid_for(8);
  if (a.gain) {
    // gain rows (QKV and gate/up inputs): the gain chunks stay in registers too
    if (chunks <= 4 * kQuantThreads)
      return launch_pdl(quant_row_cta_kernel<4, true>, grid_for(16), kQuantThreads, 0, s, a);
    if (chunks <= 8 * kQuantThreads) return launch_pdl(quant_row_cta_kernel<8, true>, grid, kQuantThreads, 0, s, a);
  } else {
    if (chunks <= 4 * kQuantThreads)
      return launch_pdl(quant_row_cta_kernel<4, false>, grid_for(16), kQuantThreads, 0, s, a);
    if (chunks <= 8 * kQuantThreads) return launch_pdl(quant_row_cta_kernel<8, false>, grid, kQuantThreads, 0, s, a);
    if (chunks <= 12 * kQuantThreads)
      return launch_pdl(quant_row_cta_kernel<12, false>, grid, kQuantThreads, 0, s, a);
    if (chunks <= 16 * kQuantThreads)
      return launch_pdl(quant_row_cta_kernel<16, false>, grid, kQuantThreads, 0, s, a);
  }
  const int64_t blocks = (a.rows + kQuantWarps - 1) / kQuantWarps;
  return launch_pdl(quant_rows_kernel, dim3(static_cast<unsigned>(blocks)), kQuantWarps * 32, 0, s, a);
}

}  // namespace svl
