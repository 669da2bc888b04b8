// Variable-length causal attention over active heads only (Sec. 3.2: a gated
// group's heads are never computed). One CTA per work item (sample, head,
// block of 64 queries); keys run from the sample's first row up to the last
// query of the block. GQA: query head h reads KV head h / (A / A_kv).
//
// Online softmax (running max and sum per row, output rescaled per key tile)
// with bf16 m16n8k16 tensor-core MMAs; K/V tiles of 64 keys are double
// buffered with cp.async; shared-memory rows are XOR-swizzled in 16-byte
// chunks so that ldmatrix is conflict-free.
#include "kernels.cuh"

namespace svl {

constexpr int kAttnThreads = 128;  // 4 warps x 16 query rows
constexpr int kKT = 64;            // keys per tile

SVL_DEVINL void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}
SVL_DEVINL void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
SVL_DEVINL void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

SVL_DEVINL void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
SVL_DEVINL void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

SVL_DEVINL void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of (row, 16-byte chunk) in a tile with DH bf16 per row.
template <int DH>
SVL_DEVINL uint32_t swz(int row, int chunk) {
  return static_cast<uint32_t>(row * DH * 2 + ((chunk ^ (row & 7)) << 4));
}

// Loads `rows` rows (row0.. of a [*, ld] bf16 matrix, column offset col0) into
// a 64 x DH tile; rows at or beyond `row_end` are zero-filled.
template <int DH>
SVL_DEVINL void load_tile(uint32_t sbase, const __nv_bfloat16* g, size_t ld, int row0, int row_end, int col0) {
  constexpr int CH = DH / 8;  // 16-byte chunks per row
  for (int i = threadIdx.x; i < 64 * CH; i += kAttnThreads) {
    const int r = i / CH, c = i % CH;
    const int gr = row0 + r;
    const bool ok = gr < row_end;
    const __nv_bfloat16* src = g + static_cast<size_t>(ok ? gr : row0) * ld + col0 + c * 8;
    cp_async16(sbase + swz<DH>(r, c), src, ok);
  }
}

template <int DH>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(AttnArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int n_items = min(*a.count, a.cap);
  if (static_cast<int>(blockIdx.x) >= n_items) return;
  const int4 it = a.items[blockIdx.x];
  const int q0 = it.x, q_end = it.y, r0 = it.z, h = it.w;
  const int kvh = h / (a.A / a.Akv);
  const size_t ldq = static_cast<size_t>(a.A) * DH, ldk = static_cast<size_t>(a.Akv) * DH;
  constexpr int TILE = 64 * DH * 2;
  const uint32_t sQ = smem_u32(smem);
  const uint32_t sK0 = sQ + TILE, sV0 = sQ + 3 * TILE;  // K: 2 buffers, V: 2 buffers, TILE apart

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kv_end = q_end;
  const int n_tiles = (kv_end - r0 + kKT - 1) / kKT;

  load_tile<DH>(sQ, a.Q, ldq, q0, q_end, h * DH);
  load_tile<DH>(sK0, a.K, ldk, r0, kv_end, kvh * DH);
  load_tile<DH>(sV0, a.V, ldk, r0, kv_end, kvh * DH);
  cp_async_commit();

  // Q fragments of this warp's 16 rows
  uint32_t qf[DH / 16][4];
  float o[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  const int g = lane >> 2, tq = lane & 3;
  const int qrow0 = q0 + warp * 16 + g;  // global query rows g and g + 8

  for (int j = 0; j < n_tiles; ++j) {
    const int buf = j & 1;
    if (j + 1 < n_tiles) {
      const int nb = buf ^ 1;
      load_tile<DH>(sK0 + nb * TILE, a.K, ldk, r0 + (j + 1) * kKT, kv_end, kvh * DH);
      load_tile<DH>(sV0 + nb * TILE, a.V, ldk, r0 + (j + 1) * kKT, kv_end, kvh * DH);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (j == 0) {
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk) {
        const int row = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int chunk = kk * 2 + (lane >> 4);
        ldsm_x4(sQ + swz<DH>(row, chunk), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    const uint32_t sK = sK0 + buf * TILE, sV = sV0 + buf * TILE;

    // S = Q K^T for 64 keys: 8 n-blocks of 8 keys
    float s[8][4];
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) s[nb][0] = s[nb][1] = s[nb][2] = s[nb][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
#pragma unroll
      for (int nb2 = 0; nb2 < 4; ++nb2) {  // two n-blocks per ldmatrix.x4
        const int key = nb2 * 16 + (lane & 7) + (lane >> 4) * 8;
        const int chunk = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sK + swz<DH>(key, chunk), b0, b1, b2, b3);
        mma16816(s[2 * nb2], qf[kk], b0, b1);
        mma16816(s[2 * nb2 + 1], qf[kk], b2, b3);
      }
    }
    // causal mask and scale (log2 domain)
    const int key_base = r0 + j * kKT;
    float mx[2] = {m_run[0], m_run[1]};
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = key_base + nb * 8 + tq * 2 + (e & 1);
        const int qr = qrow0 + (e >> 1) * 8;
        float v = s[nb][e] * a.scale_log2;
        if (key > qr || key >= kv_end) v = -INFINITY;
        s[nb][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    float corr[2], rs[2] = {0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      corr[r] = (m_run[r] == -INFINITY) ? 0.f : exp2f(m_run[r] - mx[r]);
      m_run[r] = mx[r];
    }
    const float mref0 = mx[0] == -INFINITY ? 0.f : mx[0];
    const float mref1 = mx[1] == -INFINITY ? 0.f : mx[1];
    uint32_t pf[4][4];  // P as A fragments: 4 k-steps of 16 keys
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
      const float p0 = exp2f(s[nb][0] - mref0), p1 = exp2f(s[nb][1] - mref0);
      const float p2 = exp2f(s[nb][2] - mref1), p3 = exp2f(s[nb][3] - mref1);
      rs[0] += p0 + p1;
      rs[1] += p2 + p3;
      pf[nb >> 1][(nb & 1) * 2 + 0] = pack_bf16x2(p0, p1);
      pf[nb >> 1][(nb & 1) * 2 + 1] = pack_bf16x2(p2, p3);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 1);
      rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 2);
      l_run[r] = l_run[r] * corr[r] + rs[r];
    }
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) {
      o[i][0] *= corr[0];
      o[i][1] *= corr[0];
      o[i][2] *= corr[1];
      o[i][3] *= corr[1];
    }
    // O += P V: k = 64 keys (4 steps), n = DH dims (DH/8 blocks)
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int nb2 = 0; nb2 < DH / 16; ++nb2) {
        const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int chunk = nb2 * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sV + swz<DH>(key, chunk), b0, b1, b2, b3);
        mma16816(o[2 * nb2], pf[kk], b0, b1);
        mma16816(o[2 * nb2 + 1], pf[kk], b2, b3);
      }
    }
    __syncthreads();
  }

  // normalise and store rows < q_end
  const float inv0 = l_run[0] > 0.f ? 1.f / l_run[0] : 0.f;
  const float inv1 = l_run[1] > 0.f ? 1.f / l_run[1] : 0.f;
  __nv_bfloat16* out = a.O + static_cast<size_t>(h) * DH;
#pragma unroll
  for (int nb = 0; nb < DH / 8; ++nb) {
    const int col = nb * 8 + tq * 2;
    if (qrow0 < q_end)
      *reinterpret_cast<uint32_t*>(out + static_cast<size_t>(qrow0) * ldq + col) =
          pack_bf16x2(o[nb][0] * inv0, o[nb][1] * inv0);
    if (qrow0 + 8 < q_end)
      *reinterpret_cast<uint32_t*>(out + static_cast<size_t>(qrow0 + 8) * ldq + col) =
          pack_bf16x2(o[nb][2] * inv1, o[nb][3] * inv1);
  }
}

template <int DH>
static void launch_dh(const AttnArgs& a, cudaStream_t s) {
  constexpr int smem = 5 * 64 * DH * 2;
  static bool configured = false;
  if (!configured) {
    cudaFuncSetAttribute(attn_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    configured = true;
  }
  if (a.cap > 0) attn_kernel<DH><<<a.cap, kAttnThreads, smem, s>>>(a);
}

void launch_attention(const AttnArgs& a, cudaStream_t s) {
  if (a.dh == 128) launch_dh<128>(a, s);
  else launch_dh<64>(a, s);
}

}  // namespace svl
