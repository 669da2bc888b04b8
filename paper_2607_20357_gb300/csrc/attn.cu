// Variable-length causal attention over active heads only (Sec. 3.2: the
// heads of a gated-off group are never computed), on tcgen05 tensor cores.
//
// Persistent kernel, one CTA per SM, work items (sample, active head, block
// of 128 queries) from the device schedule. Per item and per tile of 128 keys:
//   S = Q K^T          tcgen05.mma M=128 N=128 K=d_head, into one of two TMEM
//                      S buffers (S(j+1) is computed while row j's softmax runs)
//   softmax            four warps, one query row per thread: running max and
//                      sum, P = exp2(S*scale - max) rounded to bf16 and written
//                      to shared memory in the 128-byte-swizzled K-major layout
//   O_tile = P V       tcgen05.mma M=128 N=d_head K=128 into a TMEM buffer;
//                      the thread folds it into its fp32 output row in
//                      registers: O = O*exp2(m_old - m_new) + O_tile
// V arrives transposed (V^T, keys contiguous) so that both MMA operands are
// K-major. Key tiles start at the sample's first row rounded down to a
// multiple of 8 (TMA needs a 16-byte aligned innermost coordinate); keys of
// the neighbouring sample that this pulls in are masked, like every key after
// the query (causal) or past the block's last query.
//
// Warp 0: TMA producer (Q once per item, K and V^T double buffered).
// Warp 1: TMEM allocation and the MMA-issuing thread.
// Warps 2-5: softmax and output. Every wait is bounded.
#include "kernels.cuh"

namespace svl {

constexpr int kAttnThreads = 192;
constexpr int kKeyTile = 128;

template <int DH>
struct AttnSmem {
  static constexpr int kQ = 128 * DH * 2;          // Q: DH/64 atoms of 128 rows x 128 B
  static constexpr int kK = kKeyTile * DH * 2;     // K stage
  static constexpr int kV = DH * kKeyTile * 2;     // V^T stage: 2 atoms of DH rows x 128 B
  static constexpr int kP = 128 * kKeyTile * 2;    // P buffer: 2 atoms of 128 rows x 128 B
  static constexpr int q = 0;
  static constexpr int k0 = kQ;
  static constexpr int v0 = k0 + 2 * kK;
  static constexpr int p0 = v0 + 2 * kV;
  static constexpr int bars = p0 + 2 * kP;
  static constexpr int total = bars + 256 + 1024;  // + barriers + alignment slack
};

struct AttnBars {
  uint64_t q_full, q_empty, k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], p_full, o_full[2];
};

SVL_DEVINL void attn_abort(volatile int* abort, uint32_t* status) {
  *abort = 1;
  report(status, SVL_DEV_TIMEOUT);
}

SVL_DEVINL int n_key_tiles(const int4& it) {
  const int key_base = it.z & ~7;
  return (it.y - key_base + kKeyTile - 1) / kKeyTile;
}

SVL_DEVINL float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// TMEM columns: S buffers 0 and 128, P V buffers 256 and 384.
template <int DH>
__global__ void __launch_bounds__(kAttnThreads, 1) attn_tc_kernel(const __grid_constant__ AttnTcArgs a) {
  using L = AttnSmem<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  AttnBars* bar = reinterpret_cast<AttnBars*>(sm + L::bars);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&bar->q_full, 1);
    mbar_init(&bar->q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bar->k_full[i], 1);
      mbar_init(&bar->k_empty[i], 1);
      mbar_init(&bar->v_full[i], 1);
      mbar_init(&bar->v_empty[i], 1);
      mbar_init(&bar->s_full[i], 1);
      mbar_init(&bar->o_full[i], 1);
    }
    mbar_init(&bar->p_full, 128);
    *abort = 0;
    fence_barrier_init();
    fence_proxy_async();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  pdl_wait();
  const int n_items = min(*a.count, a.cap);

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int g = 0, li = 0;
      bool ok = true;
      for (int i = blockIdx.x; i < n_items && ok; i += gridDim.x, ++li) {
        const int4 it = a.items[i];
        const int h = it.w, kvh = h / (a.A / a.Akv), key_base = it.z & ~7, nt = n_key_tiles(it);
        if (!mbar_wait(&bar->q_empty, (li & 1) ^ 1, abort)) { ok = false; break; }
        mbar_arrive_expect_tx(&bar->q_full, L::kQ);
        for (int at = 0; at < DH / 64; ++at)
          tma_load_2d(sm + L::q + at * 128 * 128, &a.mapQ, &bar->q_full, h * DH + at * 64, it.x);
        for (int j = 0; j < nt; ++j, ++g) {
          const int s = g & 1;
          const uint32_t ph = ((g >> 1) & 1) ^ 1;
          const int key0 = key_base + j * kKeyTile;
          if (!mbar_wait(&bar->k_empty[s], ph, abort)) { ok = false; break; }
          mbar_arrive_expect_tx(&bar->k_full[s], L::kK);
          for (int at = 0; at < DH / 64; ++at)
            tma_load_2d(sm + L::k0 + s * L::kK + at * kKeyTile * 128, &a.mapK, &bar->k_full[s], kvh * DH + at * 64,
                        key0);
          if (!mbar_wait(&bar->v_empty[s], ph, abort)) { ok = false; break; }
          mbar_arrive_expect_tx(&bar->v_full[s], L::kV);
          for (int at = 0; at < 2; ++at)
            tma_load_2d(sm + L::v0 + s * L::kV + at * DH * 128, &a.mapVt, &bar->v_full[s], key0 + at * 64, kvh * DH);
        }
      }
      if (!ok) attn_abort(abort, a.status);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16_f32(128, kKeyTile), id_o = idesc_bf16_f32(128, DH);
      const uint32_t sq = smem_u32(sm + L::q);
      int g = 0, li = 0;
      bool ok = true;
      // S(gg) = Q K(gg)^T into S buffer gg&1; frees the K stage when done
      auto issue_s = [&](int gg, bool last_of_item) -> bool {
        const int s = gg & 1;
        if (!mbar_wait(&bar->k_full[s], (gg >> 1) & 1, abort)) return false;
        tc_fence_after();
        const uint32_t sk = smem_u32(sm + L::k0 + s * L::kK);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (128 * 128) + (kk & 3) * 32;
          const uint32_t offk = (kk >> 2) * (kKeyTile * 128) + (kk & 3) * 32;
          tc_mma_bf16(tmem + s * 128, smem_desc_sw128(sq + off), smem_desc_sw128(sk + offk), id_s, kk > 0);
        }
        tc_commit(&bar->s_full[s]);
        tc_commit(&bar->k_empty[s]);
        if (last_of_item) tc_commit(&bar->q_empty);  // Q may be replaced once these finish
        return true;
      };
      for (int i = blockIdx.x; i < n_items && ok; i += gridDim.x, ++li) {
        const int nt = n_key_tiles(a.items[i]);
        if (!mbar_wait(&bar->q_full, li & 1, abort)) { ok = false; break; }
        tc_fence_after();
        ok = issue_s(g, nt == 1) && (nt < 2 || issue_s(g + 1, nt == 2));
        for (int j = 0; j < nt && ok; ++j) {
          const int gj = g + j, s = gj & 1;
          if (!mbar_wait(&bar->p_full, gj & 1, abort) || !mbar_wait(&bar->v_full[s], (gj >> 1) & 1, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sp = smem_u32(sm + L::p0 + s * L::kP);
          const uint32_t sv = smem_u32(sm + L::v0 + s * L::kV);
#pragma unroll
          for (int kk = 0; kk < kKeyTile / 16; ++kk) {
            const uint32_t offp = (kk >> 2) * (128 * 128) + (kk & 3) * 32;
            const uint32_t offv = (kk >> 2) * (DH * 128) + (kk & 3) * 32;
            tc_mma_bf16(tmem + 256 + s * 128, smem_desc_sw128(sp + offp), smem_desc_sw128(sv + offv), id_o, kk > 0);
          }
          tc_commit(&bar->o_full[s]);
          tc_commit(&bar->v_empty[s]);
          if (j + 2 < nt) ok = issue_s(gj + 2, j + 2 == nt - 1);
        }
        g += nt;
      }
      if (!ok) attn_abort(abort, a.status);
    }
  } else {
    // ------------------------------------------------------------ softmax + output
    const int q = warp & 3;
    const int row = q * 32 + lane;  // query row within the block = TMEM lane
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const float sc = a.scale_log2;
    int g = 0;
    bool ok = true;
    for (int i = blockIdx.x; i < n_items && ok; i += gridDim.x) {
      const int4 it = a.items[i];
      const int qg = it.x + row;  // global query row
      const int key_base = it.z & ~7, nt = n_key_tiles(it);
      float o[DH];
#pragma unroll
      for (int d = 0; d < DH; ++d) o[d] = 0.f;
      float m_run = -INFINITY, l_run = 0.f;
      float cr0 = 0.f, cr1 = 0.f;  // correction factors of the (even, odd) tiles whose P V is pending

      // O = O * corr(t) + (P V)(t), once the MMA for tile t has finished
      auto fold = [&](int t) -> bool {
        const int s = t & 1;
        const bool got = mbar_wait(&bar->o_full[s], (t >> 1) & 1, abort);
        __syncwarp();
        if (!__all_sync(0xffffffffu, got)) return false;
        tc_fence_after();
        const float c = ((t - g) & 1) ? cr1 : cr0;
        float v[32];
#pragma unroll
        for (int cc = 0; cc < DH; cc += 32) {
          tmem_ld32(tmem + 256 + s * 128 + lane_off + cc, v);
#pragma unroll
          for (int e = 0; e < 32; ++e) o[cc + e] = fmaf(o[cc + e], c, v[e]);
        }
        tc_fence_before();
        return true;
      };

      for (int j = 0; j < nt; ++j) {
        const int gj = g + j, s = gj & 1;
        if (j >= 2 && !fold(gj - 2)) { ok = false; break; }
        const bool got = mbar_wait(&bar->s_full[s], (gj >> 1) & 1, abort);
        __syncwarp();
        if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
        tc_fence_after();
        const uint32_t ts = tmem + s * 128 + lane_off;
        const int kbase = key_base + j * kKeyTile;
        // keys kbase + [lo, hi) are valid for this row; a tile wholly inside
        // the sample and before the block's first query needs no mask
        const bool full = kbase >= it.z && kbase + kKeyTile - 1 <= it.x;
        const int lo = full ? 0 : max(it.z - kbase, 0);
        // (a row that precedes the whole tile has no valid key: empty range)
        const int hi = full ? kKeyTile : max(min(min(qg + 1, it.y) - kbase, kKeyTile), lo);
        float v[32];
        float mx = -INFINITY;
        for (int c = 0; c < kKeyTile; c += 32) {
          tmem_ld32(ts + c, v);
          if (full) {
#pragma unroll
            for (int e = 0; e < 32; ++e) mx = fmaxf(mx, v[e]);
          } else {
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (static_cast<unsigned>(c + e - lo) < static_cast<unsigned>(hi - lo)) mx = fmaxf(mx, v[e]);
          }
        }
        const float m_new = fmaxf(m_run, mx * sc);
        const float mref = (m_new == -INFINITY) ? 0.f : m_new;
        const float corr = (m_run == -INFINITY) ? 0.f : ex2(m_run - mref);
        m_run = m_new;
        if (j & 1) cr1 = corr; else cr0 = corr;
        uint8_t* prow = sm + L::p0 + s * L::kP + row * 128;
        float rs = 0.f;
        for (int c = 0; c < kKeyTile; c += 32) {
          tmem_ld32(ts + c, v);
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float x0 = fmaf(v[e], sc, -mref), x1 = fmaf(v[e + 1], sc, -mref);
            if (!full) {
              if (static_cast<unsigned>(c + e - lo) >= static_cast<unsigned>(hi - lo)) x0 = -INFINITY;
              if (static_cast<unsigned>(c + e + 1 - lo) >= static_cast<unsigned>(hi - lo)) x1 = -INFINITY;
            }
            const float p0 = ex2(x0), p1 = ex2(x1);
            rs += p0 + p1;
            pk[e >> 1] = pack_bf16x2(p0, p1);
          }
          // keys c..c+31: atom c/64, 16-byte chunks (c%64)/8 .. +3, 128-byte swizzle
          const int atom = c >> 6, ch0 = (c & 63) >> 3;
          uint8_t* base = prow + atom * (128 * 128);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int ch = (ch0 + u) ^ (row & 7);
            *reinterpret_cast<uint4*>(base + (ch << 4)) =
                make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
          }
        }
        l_run = l_run * corr + rs;
        fence_proxy_async();  // P written by threads, read by the tensor core
        tc_fence_before();
        mbar_arrive(&bar->p_full);
      }
      if (ok && nt >= 2) ok = fold(g + nt - 2);
      if (ok) ok = fold(g + nt - 1);
      g += nt;
      if (!ok) break;
      if (qg < it.y) {
        const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
        uint4* dst = reinterpret_cast<uint4*>(a.O + static_cast<size_t>(qg) * a.ldo + static_cast<size_t>(it.w) * DH);
#pragma unroll
        for (int d = 0; d < DH; d += 8)
          dst[d / 8] = make_uint4(pack_bf16x2(o[d] * inv, o[d + 1] * inv), pack_bf16x2(o[d + 2] * inv, o[d + 3] * inv),
                                  pack_bf16x2(o[d + 4] * inv, o[d + 5] * inv), pack_bf16x2(o[d + 6] * inv, o[d + 7] * inv));
      }
    }
    if (!ok) attn_abort(abort, a.status);
  }

  __syncwarp();
  if (*abort) {
    long long t0 = clock64();
    while (clock64() - t0 < 20000000LL) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int DH>
static cudaError_t launch_dh(const AttnTcArgs& a, int grid, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         AttnSmem<DH>::total);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  return launch_pdl(attn_tc_kernel<DH>, grid, kAttnThreads, AttnSmem<DH>::total, s, a);
}

cudaError_t launch_attention_tc(const AttnTcArgs& a, int grid, cudaStream_t s) {
  if (a.cap <= 0) return cudaSuccess;
  return a.dh == 128 ? launch_dh<128>(a, grid, s) : launch_dh<64>(a, grid, s);
}

}  // namespace svl
