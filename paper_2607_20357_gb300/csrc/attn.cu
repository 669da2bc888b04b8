// Variable-length causal attention over active heads only (Sec. 3.2: the
// heads of a gated-off group are never computed), on tcgen05 tensor cores.
//
// Persistent kernel, one CTA per SM, two independent query-block pipelines
// ("slots") per CTA. A unit of work is one block of up to 128 queries of one
// (sample, active head); every item of the device schedule (up to 256
// queries) gives two units, its two 128-query halves, later half first. The
// schedule lists one head's items next to each other, latest first, and each
// slot takes the next unit from a counter in global memory when it is ready
// for one: the units of a head run at about the same time on several SMs and
// share its keys and values in L2, the heaviest units start first, and no
// slot idles while units are left. Neither slot ever waits for the other's
// chain. Keys come in tiles of 64. Per slot and tile:
//   S = Q K^T      tcgen05.mma M=128 N=64 K=d_head into one of two S buffers
//                  in TMEM, so S of tile j+1 is computed while the softmax
//                  works on tile j;
//   softmax        one query row per thread: P = exp2(S*scale - m) rounded
//                  to bf16 and written back over the tile's own S columns in
//                  TMEM (tcgen05.st, two keys per column), row sum;
//   O += P V       tcgen05.mma M=128 N=d_head K=64 into the slot's O columns,
//                  A = P read from tensor memory, B = the V^T tile.
// P never touches shared memory, and the softmax of tile j+1 does not wait
// for the P V of tile j: the next S MMA into the same buffer is issued after
// that P V, and the tensor core executes one thread's MMAs in order.
// The running max m is the row max of the unit's first tile. Later tiles form
// P against it and only check their row sum: while it stays at most 2^14
// (every entry of P is then at most 2^14, far from any overflow) O needs no
// correction and no tile max is computed. A row whose sum exceeds that (or is
// not finite) takes the tile's max as the new m, O and the row sum are
// rescaled in place and the tile's P is formed again. O / rowsum is written
// out once per unit.
//
// V arrives transposed (V^T, keys contiguous) so that both operands are
// K-major. K and V^T tiles go through the slot's own 4-stage ring, which the
// producer fills in the order the MMA thread consumes them (K of tile j+1
// can load while tiles j-1 and j are in use). Key tiles start at the sample's
// first row rounded down to a multiple of 8 (TMA needs a 16-byte aligned
// innermost coordinate); keys of the neighbouring sample that this pulls in
// are masked, like every key after the query (causal) or past the sample's
// end. Each softmax warp writes its own 32 output rows: through its part of
// the slot's output staging buffer and a TMA tensor store per 64 columns when
// all 32 rows exist, with per-thread stores otherwise.
//
// Warps: 0 / 6 TMA producers of slot 0 / 1 (the producer also takes the
// slot's units from the counter and passes them to the other warps of the
// slot through a small ring in shared memory); 1 / 7 MMA issuers (warp 1 also
// owns the TMEM allocation: slot s uses columns 256 s .. 256 s + 255 for S0,
// S1 and O); 2-5 / 8-11 softmax and output of slot 0 / 1. Every barrier
// completes at most once ahead of its waiter; every wait is bounded.
#include "kernels.cuh"

namespace svl {

constexpr float kTileSumMax = 16384.f;  // largest row sum of a tile's P formed against the running max
static_assert(kAttnQ == 256, "an attention item is two blocks of 128 queries");

SVL_DEVINL void attn_abort(volatile int* abort, uint32_t* status) {
  *abort = 1;
  report(status, SVL_DEV_TIMEOUT);
}

SVL_DEVINL float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

SVL_DEVINL float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Two fp32 lanes in one 64-bit register: (a*b + c) and (a + b) per lane.
SVL_DEVINL uint64_t f2(float lo, float hi) {
  return (static_cast<uint64_t>(__float_as_uint(hi)) << 32) | __float_as_uint(lo);
}
SVL_DEVINL uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
SVL_DEVINL uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
SVL_DEVINL float lo2(uint64_t v) { return __uint_as_float(static_cast<uint32_t>(v)); }
SVL_DEVINL float hi2(uint64_t v) { return __uint_as_float(static_cast<uint32_t>(v >> 32)); }

// Ring positions of a unit's 2n tiles relative to its first, in the order the
// MMA thread consumes them: K(0), then per round j = 1..n: K(j) (while j < n)
// and V(j-1).
SVL_DEVINL int pos_k(int j) { return j == 0 ? 0 : 2 * j - 1; }
SVL_DEVINL int pos_v(int m, int n) { return m + 1 < n ? 2 * m + 2 : 2 * m + 1; }

// Scores outside the valid keys [lo, lo + span) of the tile set to -inf.
SVL_DEVINL void mask64(uint32_t* sv, int lo, unsigned span) {
#pragma unroll
  for (int e = 0; e < 64; ++e)
    if (static_cast<unsigned>(e - lo) >= span) sv[e] = 0xff800000u;
}

// Row max of 64 scores, in four independent chains.
SVL_DEVINL float row_max64(const uint32_t* sv) {
  float m0 = -INFINITY, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY;
#pragma unroll
  for (int e = 0; e < 64; e += 8) {
    m0 = max3(m0, __uint_as_float(sv[e]), __uint_as_float(sv[e + 1]));
    m1 = max3(m1, __uint_as_float(sv[e + 2]), __uint_as_float(sv[e + 3]));
    m2 = max3(m2, __uint_as_float(sv[e + 4]), __uint_as_float(sv[e + 5]));
    m3 = max3(m3, __uint_as_float(sv[e + 6]), __uint_as_float(sv[e + 7]));
  }
  return fmaxf(fmaxf(m0, m1), fmaxf(m2, m3));
}

// P = exp2(S*scale - m) for 64 keys (masked scores are -inf and give 0),
// rounded to bf16 and packed two keys per 32-bit word (lower key in the low
// half) into pk[32], the layout of the A operand in tensor memory; returns
// the row sum of the unrounded values.
SVL_DEVINL float exp_pack64(const uint32_t* sv, uint64_t sc2, uint64_t nm2, uint32_t* pk) {
  uint64_t acc0 = 0, acc1 = 0;
#pragma unroll
  for (int e2 = 0; e2 < 32; ++e2) {
    const int e = 2 * e2;
    const uint64_t xv = fma2(f2(__uint_as_float(sv[e]), __uint_as_float(sv[e + 1])), sc2, nm2);
    const float p0 = ex2(lo2(xv)), p1 = ex2(hi2(xv));
    if (e2 & 1) acc1 = add2(acc1, f2(p0, p1)); else acc0 = add2(acc0, f2(p0, p1));
    pk[e2] = pack_bf16x2(p0, p1);
  }
  const uint64_t acc = add2(acc0, acc1);
  return lo2(acc) + hi2(acc);
}

constexpr int kPipeThreads = 384;
constexpr int kPipeKeys = 64;
constexpr int kPipeRing = 4;
constexpr int kUnitRing = 4;   // units handed from a slot's producer to its MMA and softmax warps

template <int DH>
struct PipeSmem {
  static constexpr int kQAtom = 128 * 128;            // 128 rows x 128 B
  static constexpr int kQ = 128 * DH * 2;             // DH/64 atoms
  static constexpr int kKAtom = kPipeKeys * 128;      // 64 keys x 128 B
  static constexpr int kKV = kPipeKeys * DH * 2;      // K tile (DH/64 atoms) or V^T tile (DH rows x 128 B)
  static constexpr int kP = 128 * kPipeKeys * 2;      // output staging: 128 rows x 64 columns
  static constexpr int q0 = 0;
  static constexpr int p0 = q0 + kQ;
  static constexpr int r0 = p0 + kP;
  static constexpr int slot = r0 + kPipeRing * kKV;   // bytes per slot (multiple of 1024)
  static constexpr int bars = 2 * slot;
  static constexpr int total = bars + 1024 + 1024;
};
static_assert(PipeSmem<128>::total <= 232448, "pipelined attention shared memory");

struct PipeBars {
  uint64_t q_full, q_empty, r_full[kPipeRing], r_empty[kPipeRing], s_full[2], p_full[2], pv_done[2];
  uint64_t unit_full[kUnitRing], unit_empty[kUnitRing];
  int4 item[kUnitRing];  // the unit's schedule item
  int unit[kUnitRing];   // unit index, or -1: no units left
};
static_assert(2 * sizeof(PipeBars) + 8 <= 1024, "attention barriers");

// Unit u: half 1 - (u & 1) of item `it` = item u / 2 of the schedule (an
// item's later half first). False for an empty half (the short last item of
// a sample).
SVL_DEVINL bool unit_rows(const int4& it, int u, int& qb0, int& qend, int& ntiles) {
  const int half = (u & 1) ^ 1;
  qb0 = it.x + 128 * half;
  qend = min(qb0 + 128, it.y);
  if (qend <= qb0) return false;
  const int key_base = it.z & ~7;
  ntiles = (qend - key_base + kPipeKeys - 1) / kPipeKeys;
  return true;
}

template <int DH>
__global__ void __launch_bounds__(kPipeThreads, 1) attn_tc_kernel(const __grid_constant__ AttnTcArgs a) {
  using L = PipeSmem<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  PipeBars* bars = reinterpret_cast<PipeBars*>(sm + L::bars);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int sl = 0; sl < 2; ++sl) {
      PipeBars* b = bars + sl;
      mbar_init(&b->q_full, 1);
      mbar_init(&b->q_empty, 1);
      for (int i = 0; i < kPipeRing; ++i) {
        mbar_init(&b->r_full[i], 1);
        mbar_init(&b->r_empty[i], 1);
      }
      for (int i = 0; i < 2; ++i) {
        mbar_init(&b->s_full[i], 1);
        mbar_init(&b->p_full[i], 128);
        mbar_init(&b->pv_done[i], 1);
      }
      for (int i = 0; i < kUnitRing; ++i) {
        mbar_init(&b->unit_full[i], 1);
        mbar_init(&b->unit_empty[i], 5);  // the MMA thread and the four softmax warps
      }
    }
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
  const int n_units = 2 * n_items;
  const int group = a.A / a.Akv;
  int kunit = 0;  // units taken from (or, producer, put into) the slot's ring
  const int slot = warp < 6 ? 0 : 1;
  const int role = warp < 6 ? warp : warp - 6;  // 0 producer, 1 MMA, 2-5 softmax
  PipeBars* bar = bars + slot;
  uint8_t* ss = sm + slot * L::slot;
  const uint32_t tbase = tmem + 256 * slot;      // S0, S1 at +0, +64; O at +128

  if (role == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int g = 0, nq = 0;
      bool ok = true;
      // passes unit u (-1: none left) and its item to the MMA and softmax
      // warps of the slot
      auto post = [&](int u, const int4& it) -> bool {
        const int i = kunit % kUnitRing;
        if (!mbar_wait(&bar->unit_empty[i], ((kunit / kUnitRing) & 1) ^ 1, abort)) return false;
        bar->unit[i] = u;
        bar->item[i] = it;
        mbar_arrive(&bar->unit_full[i]);  // release: the stores above are seen by the waiters
        ++kunit;
        return true;
      };
      // the next non-empty unit from the counter (u >= n_units: none left)
      auto take = [&](int& u, int4& it, int& qb0, int& qend, int& n) {
        for (;;) {
          u = atomicAdd(a.next_unit, 1);
          if (u >= n_units) return;
          it = a.items[u >> 1];
          if (unit_rows(it, u, qb0, qend, n)) return;
        }
      };
      int u, qb0 = 0, qend = 0, n = 0;
      int4 it = make_int4(0, 0, 0, 0);
      take(u, it, qb0, qend, n);
      while (ok) {
        if (!post(u < n_units ? u : -1, it)) { ok = false; break; }
        if (u >= n_units) break;
        const int kvh = it.w / group, key_base = it.z & ~7;
        if (!mbar_wait(&bar->q_empty, (nq & 1) ^ 1, abort)) { ok = false; break; }
        ++nq;
        mbar_arrive_expect_tx(&bar->q_full, L::kQ);
        for (int at = 0; at < DH / 64; ++at)
          tma_load_2d(ss + L::q0 + at * L::kQAtom, &a.mapQ, &bar->q_full, it.w * DH + at * 64, qb0);
        for (int p = 0; p < 2 * n && ok; ++p, ++g) {
          const bool is_k = p == 0 || (p & 1 && p < 2 * n - 1);
          const int tile = is_k ? (p + 1) >> 1 : (p == 2 * n - 1 ? n - 1 : (p >> 1) - 1);
          const int st = g % kPipeRing;
          if (!mbar_wait(&bar->r_empty[st], ((g / kPipeRing) & 1) ^ 1, abort)) { ok = false; break; }
          mbar_arrive_expect_tx(&bar->r_full[st], L::kKV);
          uint8_t* dst = ss + L::r0 + st * L::kKV;
          const int key0 = key_base + tile * kPipeKeys;
          if (is_k) {
            for (int at = 0; at < DH / 64; ++at)
              tma_load_2d(dst + at * L::kKAtom, &a.mapK64, &bar->r_full[st], kvh * DH + at * 64, key0);
          } else {
            tma_load_2d(dst, &a.mapVt, &bar->r_full[st], key0, kvh * DH);
          }
        }
        // the next unit, taken while this one's tiles are in flight
        if (ok) take(u, it, qb0, qend, n);
      }
      if (!ok) attn_abort(abort, a.status);
    }
  } else if (role == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16_f32(128, kPipeKeys), id_o = idesc_bf16_f32(128, DH);
      int g = 0, nq = 0, t = 0;  // ring position, units, tiles so far
      bool ok = true;
      auto ring_wait = [&](int pos) -> bool {
        if (!mbar_wait(&bar->r_full[pos % kPipeRing], (pos / kPipeRing) & 1, abort)) return false;
        tc_fence_after();
        return true;
      };
      auto mma_s = [&](int b, int pos) {
        const uint64_t dq = smem_desc_sw128(smem_u32(ss + L::q0));
        const uint64_t dk = smem_desc_sw128(smem_u32(ss + L::r0 + (pos % kPipeRing) * L::kKV));
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t offq = ((kk >> 2) * L::kQAtom + (kk & 3) * 32) >> 4;
          const uint32_t offk = ((kk >> 2) * L::kKAtom + (kk & 3) * 32) >> 4;
          tc_mma_bf16(tbase + 64 * b, dq + offq, dk + offk, id_s, kk > 0);
        }
        tc_commit(&bar->s_full[b]);
      };
      auto mma_pv = [&](int b, int pos, bool acc) {
        // P of this tile: 32 columns of packed bf16 over its S buffer
        const uint64_t dv = smem_desc_sw128(smem_u32(ss + L::r0 + (pos % kPipeRing) * L::kKV));
#pragma unroll
        for (int kk = 0; kk < kPipeKeys / 16; ++kk)
          tc_mma_bf16_ts(tbase + 128, tbase + 64 * b + 8 * kk, dv + ((kk * 32) >> 4), id_o, (acc || kk > 0) ? 1u : 0u);
        tc_commit(&bar->pv_done[b]);
      };
      while (ok) {
        const int i = kunit % kUnitRing;
        ok = mbar_wait(&bar->unit_full[i], (kunit / kUnitRing) & 1, abort);
        if (!ok) break;
        const int u = *reinterpret_cast<volatile int*>(&bar->unit[i]);
        const int4 it = bar->item[i];  // after the acquiring wait (the asm is a compiler barrier)
        mbar_arrive(&bar->unit_empty[i]);
        ++kunit;
        if (u < 0) break;
        int qb0, qend, n;
        unit_rows(it, u, qb0, qend, n);
        ok = mbar_wait(&bar->q_full, nq & 1, abort);
        ++nq;
        if (!ok) break;
        tc_fence_after();
        // S of tile 0
        ok = ring_wait(g + pos_k(0));
        if (!ok) break;
        mma_s(t & 1, g + pos_k(0));
        if (n == 1) tc_commit(&bar->q_empty);
        tc_commit(&bar->r_empty[(g + pos_k(0)) % kPipeRing]);
        for (int j = 0; j < n && ok; ++j) {
          if (j + 1 < n) {
            // its S buffer held P of tile t+j-1, read by the P V issued
            // (after p_full) in the previous round: in-order MMAs
            const int gk = g + pos_k(j + 1);
            ok = ring_wait(gk);
            if (!ok) break;
            mma_s((t + j + 1) & 1, gk);
            if (j + 1 == n - 1) tc_commit(&bar->q_empty);
            tc_commit(&bar->r_empty[gk % kPipeRing]);
          }
          const int tj = t + j;
          ok = mbar_wait(&bar->p_full[tj & 1], (tj >> 1) & 1, abort);
          if (!ok) break;
          tc_fence_after();
          const int gv = g + pos_v(j, n);
          ok = ring_wait(gv);
          if (!ok) break;
          mma_pv(tj & 1, gv, j > 0);
          tc_commit(&bar->r_empty[gv % kPipeRing]);
        }
        t += n;
        g += 2 * n;
      }
      if (!ok) attn_abort(abort, a.status);
    }
  } else {
    // ------------------------------------------------------------ softmax + output
    const int q = warp & 3;         // TMEM lane quarter this warp may access
    const int row = q * 32 + lane;  // query row within the block = TMEM lane
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const uint32_t t_o = tbase + 128 + lane_off;
    const float sc = a.scale_log2;
    const uint64_t sc2 = f2(sc, sc);
    int t = 0;
    bool ok = true;
    auto wait_all = [&](uint64_t* b, uint32_t parity) -> bool {
      const bool got = mbar_wait(b, parity, abort);
      __syncwarp();
      return __all_sync(0xffffffffu, got);
    };
    while (ok) {
      const int i = kunit % kUnitRing;
      if (!wait_all(&bar->unit_full[i], (kunit / kUnitRing) & 1)) { ok = false; break; }
      const int u = *reinterpret_cast<volatile int*>(&bar->unit[i]);
      const int4 it = bar->item[i];  // after the acquiring wait (the asm is a compiler barrier)
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->unit_empty[i]);
      ++kunit;
      if (u < 0) break;
      int qb0, qend, n;
      unit_rows(it, u, qb0, qend, n);
      const int qg = qb0 + row;
      const int key_base = it.z & ~7;
      float m_run = -INFINITY, l_run = 0.f;
      // a warp whose 32 rows all lie past the block's end (the short last
      // block of a sample) only keeps the tile barriers in step: its rows of
      // S, P and O are never stored, and the MMA rows are independent
      const bool idle = qb0 + q * 32 >= qend;
      for (int j = 0; j < n; ++j, ++t) {
        const int b = t & 1;
        if (!wait_all(&bar->s_full[b], (t >> 1) & 1)) { ok = false; break; }
        if (idle) {
          mbar_arrive(&bar->p_full[b]);
          continue;
        }
        tc_fence_after();
        const int kbase = key_base + j * kPipeKeys;
        const bool full = kbase >= it.z && kbase + kPipeKeys - 1 <= qb0;
        const int lo = full ? 0 : max(it.z - kbase, 0);
        const int hi = full ? kPipeKeys : max(min(min(qg + 1, qend) - kbase, kPipeKeys), lo);
        const unsigned span = static_cast<unsigned>(hi - lo);
        uint32_t sv[64];
        tmem_ld32_async(tbase + 64 * b + lane_off, sv);
        tmem_ld32_async(tbase + 64 * b + 32 + lane_off, sv + 32);
        tmem_ld_wait32(sv);
        tmem_ld_wait32(sv + 32);
        if (!full) mask64(sv, lo, span);
        if (j == 0) m_run = row_max64(sv) * sc;
        uint32_t pk[32];
        float l_tile = exp_pack64(sv, sc2, f2(m_run == -INFINITY ? 0.f : -m_run, m_run == -INFINITY ? 0.f : -m_run), pk);
        const bool need = !(l_tile <= kTileSumMax);  // also true for inf / NaN
        if (__any_sync(0xffffffffu, need)) {
          // a row of this tile grew past the running max: move it to the
          // tile's max, rescale the row's O and sum, form P again
          float corr = 1.f;
          if (need) {
            const float m_tile = row_max64(sv) * sc;
            if (m_tile > m_run) {
              corr = ex2(m_run - m_tile);
              l_run *= corr;
              m_run = m_tile;
            }
          }
          if (j > 0) {
            // O must hold P V of every earlier tile before it is rescaled
            if (!wait_all(&bar->pv_done[(t - 1) & 1], ((t - 1) >> 1) & 1)) { ok = false; break; }
            tc_fence_after();
#pragma unroll 1
            for (int cc = 0; cc < DH; cc += 32) {
              uint32_t ov[32];
              tmem_ld32_async(t_o + cc, ov);
              tmem_ld_wait32(ov);
#pragma unroll
              for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * corr);
              tmem_st32(t_o + cc, ov);
            }
            tmem_st_wait();
          }
          const float mref = m_run == -INFINITY ? 0.f : m_run;
          l_tile = exp_pack64(sv, sc2, f2(-mref, -mref), pk);
        }
        l_run += l_tile;
        // P over the first 32 columns of this tile's S buffer (its S values
        // are in registers already)
        tmem_st32(tbase + 64 * b + lane_off, pk);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&bar->p_full[b]);
      }
      if (!ok) break;
      if (idle) continue;  // no rows of this warp to write
      // block done: O of the last P V, divided by the row sum
      if (!wait_all(&bar->pv_done[(t - 1) & 1], ((t - 1) >> 1) & 1)) { ok = false; break; }
      tc_fence_after();
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      const int wrow0 = q * 32;  // this warp's first row in the block
      if (qb0 + wrow0 + 32 <= qend) {
        // all 32 rows exist: 64 columns at a time into this warp's rows of the
        // staging buffer (swizzled like a TMA box), one TMA store each by lane 0
        uint8_t* prow = ss + L::p0 + row * 128;
#pragma unroll 1
        for (int h = 0; h < DH / 64; ++h) {
          uint32_t ov[64];
          tmem_ld32_async(t_o + 64 * h, ov);
          tmem_ld32_async(t_o + 64 * h + 32, ov + 32);
          // the previous store from these rows (this unit's or the last one's)
          // has left shared memory
          if (lane == 0) bulk_wait_read0();
          __syncwarp();
          tmem_ld_wait32(ov);
          tmem_ld_wait32(ov + 32);
#pragma unroll
          for (int d = 0; d < 64; d += 8) {
            const int chunk = d / 8;  // 16-byte chunk of the 128-byte row
            *reinterpret_cast<uint4*>(prow + ((chunk ^ (row & 7)) << 4)) = make_uint4(
                pack_bf16x2(__uint_as_float(ov[d]) * inv, __uint_as_float(ov[d + 1]) * inv),
                pack_bf16x2(__uint_as_float(ov[d + 2]) * inv, __uint_as_float(ov[d + 3]) * inv),
                pack_bf16x2(__uint_as_float(ov[d + 4]) * inv, __uint_as_float(ov[d + 5]) * inv),
                pack_bf16x2(__uint_as_float(ov[d + 6]) * inv, __uint_as_float(ov[d + 7]) * inv));
          }
          fence_proxy_async();  // generic-proxy writes, read by the TMA unit
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&a.mapO, ss + L::p0 + wrow0 * 128, it.w * DH + 64 * h, qb0 + wrow0);
            bulk_commit();
          }
        }
      } else {
        uint4* dst = reinterpret_cast<uint4*>(a.O + static_cast<size_t>(qg) * a.ldo + static_cast<size_t>(it.w) * DH);
#pragma unroll 1
        for (int cc = 0; cc < DH; cc += 32) {
          uint32_t ov[32];
          tmem_ld32_async(t_o + cc, ov);
          tmem_ld_wait32(ov);
          if (qg < qend) {
#pragma unroll
            for (int d = 0; d < 32; d += 8)
              dst[(cc + d) / 8] = make_uint4(
                  pack_bf16x2(__uint_as_float(ov[d]) * inv, __uint_as_float(ov[d + 1]) * inv),
                  pack_bf16x2(__uint_as_float(ov[d + 2]) * inv, __uint_as_float(ov[d + 3]) * inv),
                  pack_bf16x2(__uint_as_float(ov[d + 4]) * inv, __uint_as_float(ov[d + 5]) * inv),
                  pack_bf16x2(__uint_as_float(ov[d + 6]) * inv, __uint_as_float(ov[d + 7]) * inv));
          }
        }
      }
      tc_fence_before();  // O read before the next unit's first P V overwrites it
    }
    if (lane == 0) bulk_wait0();  // this warp's output stores are complete
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
static cudaError_t launch_pipe(const AttnTcArgs& a, int grid, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         PipeSmem<DH>::total);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  return launch_pdl(attn_tc_kernel<DH>, grid, kPipeThreads, PipeSmem<DH>::total, s, a);
}

cudaError_t launch_attention_tc(const AttnTcArgs& a, int grid, cudaStream_t s) {
  if (a.cap <= 0) return cudaSuccess;
  return a.dh == 128 ? launch_pipe<128>(a, grid, s) : launch_pipe<64>(a, grid, s);
}

}  // namespace svl
