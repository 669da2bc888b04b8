// Persistent warp-specialised tcgen05 GEMM with fused epilogues (sm_103a).
//
//   warp 0      one thread issues TMA loads of A (128 rows x 128 bytes) and B
//               (up to 2 x 128 rows x 128 bytes) per stage into a 4-stage
//               shared-memory ring: 64 K of bf16 or 128 K of e4m3;
//   warp 1      allocates 512 TMEM columns; one thread issues
//               tcgen05.mma (M = 128, N <= 256, K = 16 per bf16 instruction,
//               32 per e4m3 one) and commits stage releases and
//               accumulator-ready signals;
//   warps 2-5   epilogue: tcgen05.ld of their 32-lane quarter of the
//               accumulator, fused math, global stores. Two accumulators
//               alternate so the epilogue of tile i overlaps tile i+1.
//
// Every wait is bounded (kWaitCycles); a time-out sets SVL_DEV_TIMEOUT in the
// status word, stops all roles, lets in-flight copies land, frees TMEM and
// returns.
#include "gemm.cuh"

namespace svl {

struct TileInfo {
  int m0, m_end, n0, ncols, mat, kmask;
  int part, nsplit, slot;  // K-split share (nsplit == 1: the whole tile)
  bool valid;
};

SVL_DEVINL int num_tiles(const GemmParams& p) {
  if (p.tiles) {
    int n = *p.tile_count;
    return n < 0 ? 0 : (n > p.max_tiles ? p.max_tiles : n);
  }
  return p.grid_m * p.grid_n;
}

SVL_DEVINL TileInfo get_tile(const GemmParams& p, int t) {
  TileInfo ti;
  if (p.tiles) {
    int4 v = p.tiles[t];
    ti.m0 = v.x;
    ti.m_end = v.y;
    ti.n0 = v.z;
    ti.ncols = tile_ncols(v.w);
    ti.mat = tile_mat(v.w);
    ti.kmask = tile_kmask(v.w);
    ti.valid = ti.ncols > 0 && ti.m_end > ti.m0 && ti.mat < 3;
  } else {
    int mi = t % p.grid_m, ni = t / p.grid_m;
    int mlim = p.m_limit;
    if (p.m_limit_dev) mlim = min(mlim, *p.m_limit_dev);
    ti.m0 = mi * kBM;
    ti.m_end = min(ti.m0 + kBM, mlim);
    ti.n0 = ni * p.bn;
    ti.ncols = min(p.bn, p.n_limit - ti.n0);
    ti.mat = 0;
    ti.kmask = 0;
    ti.valid = ti.m0 < mlim && ti.ncols > 0;
  }
  ti.part = 0;
  ti.nsplit = 1;
  ti.slot = 0;
  if (p.ks_info && t >= p.ks_info[0]) {
    const int r = p.ks_info[1], sp = p.ks_info[2];
    if (r > 0 && sp > 1) {
      const int u = t - p.ks_info[0];
      ti.slot = u % r;
      ti.part = u / r;
      ti.nsplit = sp;
    }
  }
  return ti;
}

// Share [i0, i1) of the tile's active K blocks (all of them unless K-split).
SVL_DEVINL void k_share(const TileInfo& ti, int nkb, int kgb, int& i0, int& i1) {
  const int n = ti.kmask ? __popc(ti.kmask) * kgb : nkb;
  i0 = (n * ti.part) / ti.nsplit;
  i1 = (n * (ti.part + 1)) / ti.nsplit;
}

// Walks the K blocks of a tile, skipping the blocks of gated-off groups
// (kmask bit j clear: K blocks [j*kgb, (j+1)*kgb) are not visited). The group
// index is kept incrementally: no division in the issue loops.
struct KWalk {
  int kb, grp, kin;
  const int nkb, kgb, kmask;
  SVL_DEVINL KWalk(int nkb_, int kgb_, int kmask_) : kb(-1), grp(0), kin(-1), nkb(nkb_), kgb(kgb_), kmask(kmask_) {}
  // advances to the next active K block; false when the tile is done
  SVL_DEVINL bool next() {
    while (true) {
      ++kb;
      if (kb >= nkb) return false;
      if (++kin == kgb) {
        kin = 0;
        ++grp;
      }
      if (kmask == 0 || ((kmask >> grp) & 1)) return true;
    }
  }
};

SVL_DEVINL void set_abort(volatile int* abort, uint32_t* status) {
  *abort = 1;
  report(status, SVL_DEV_TIMEOUT);
}

// Stage geometry per epilogue: the token-score GEMM streams the features
// once and reads a B box of only H rows per stage (H <= 64: 24 KB stages,
// nine deep; H <= 128: 32 KB, six deep), keeping more feature bytes in flight.
// THIN launches (at most kThinRows rows of A, e.g. one row per sample in
// decode) are weight-streaming: their A box is kThinRows rows, so a stage is
// 36 KB and six of them keep 192 KB of weights in flight per SM. The MMA
// still reads 128 rows of A; rows past kThinRows come from the B tile that
// follows in the stage and only reach accumulator rows that are never stored.
template <int KIND, bool THIN = false>
struct StageCfg {
  static constexpr int stages = kStages;
  static constexpr int abytes = kABytes;
  static constexpr int bytes = kStageBytes;
};
template <int KIND>
struct StageCfg<KIND, true> {
  static constexpr int stages = 6;
  static constexpr int abytes = kThinRows * 128;
  static constexpr int bytes = abytes + 2 * kBHalfBytes;
};
template <>
struct StageCfg<EPI_SCORE, false> {
  static constexpr int stages = 9;
  static constexpr int abytes = kABytes;
  static constexpr int bytes = kABytes + kBHalfBytes / 2;
};
template <>
struct StageCfg<EPI_SCORE_WIDE, false> {
  static constexpr int stages = 6;
  static constexpr int abytes = kABytes;
  static constexpr int bytes = kABytes + kBHalfBytes;
};

// ------------------------------------------------------------------ producer
template <int NST, int SBYTES, int ABYTES, bool F8>
SVL_DEVINL void producer_loop(const GemmParams& p, uint8_t* stages, uint64_t* full,
                              uint64_t* empty, volatile int* abort) {
  constexpr int BK = F8 ? kBK8 : kBK;
  const int ntiles = num_tiles(p);
  const int nkb = p.K / BK, kgb = p.kgroup / BK;
  const uint64_t pol = l2_evict_first_policy();
  int s = 0;
  uint32_t ph = 0;
  for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
    TileInfo ti = get_tile(p, t);
    if (!ti.valid) continue;
    const int halves = p.b_split ? 2 : (ti.ncols > kBHalf ? 2 : 1);
    const CUtensorMap* mb0 = p.b_split ? &p.mapB[0] : &p.mapB[ti.mat];
    const CUtensorMap* mb1 = p.b_split ? &p.mapB[1] : &p.mapB[ti.mat];
    const int y1 = p.b_split ? ti.n0 : ti.n0 + kBHalf;
    const uint32_t bytes = ABYTES + halves * (p.b_box_rows ? p.b_box_rows * 128 : kBHalfBytes);
    KWalk w(nkb, kgb, ti.kmask);
    int i0, i1;
    k_share(ti, nkb, kgb, i0, i1);
    for (int i = 0; i < i0; ++i) w.next();
    for (int i = i0; i < i1; ++i) {
      w.next();
      const int kb = w.kb;
      if (!mbar_wait(&empty[s], ph ^ 1, abort)) {
        set_abort(abort, p.status);
        return;
      }
      uint8_t* sa = stages + s * SBYTES;
      uint8_t* sb = sa + ABYTES;
      mbar_arrive_expect_tx(&full[s], bytes);
      if (p.a_evict_first)
        tma_load_2d_hint(sa, &p.mapA, &full[s], kb * BK, ti.m0, pol);
      else
        tma_load_2d(sa, &p.mapA, &full[s], kb * BK, ti.m0);
      tma_load_2d(sb, mb0, &full[s], kb * BK, ti.n0);
      if (halves == 2) tma_load_2d(sb + kBHalfBytes, mb1, &full[s], kb * BK, y1);
      if (++s == NST) {
        s = 0;
        ph ^= 1;
      }
    }
  }
}

// ------------------------------------------------------------------ MMA issuer
template <int NST, int SBYTES, int ABYTES, bool F8>
SVL_DEVINL void mma_loop(const GemmParams& p, uint8_t* stages, uint64_t* full, uint64_t* empty,
                         uint64_t* tfull, uint64_t* tempty, uint32_t tmem, volatile int* abort) {
  constexpr int BK = F8 ? kBK8 : kBK;
  const int ntiles = num_tiles(p);
  const int nkb = p.K / BK, kgb = p.kgroup / BK;
  int s = 0, it = 0;
  uint32_t ph = 0;
  for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
    TileInfo ti = get_tile(p, t);
    if (!ti.valid) continue;
    const int acc = it & 1;
    const uint32_t aph = (it >> 1) & 1;
    if (!mbar_wait(&tempty[acc], aph ^ 1, abort)) {
      set_abort(abort, p.status);
      return;
    }
    tc_fence_after();
    const int n = p.b_split ? 2 * kBHalf : ((ti.ncols + 15) & ~15);
    const uint32_t idesc = F8 ? idesc_e4m3_f32(kBM, n) : idesc_bf16_f32(kBM, n);
    const uint32_t d = tmem + acc * kAccCols;
    uint32_t accumulate = 0;
    int i0, i1;
    k_share(ti, nkb, kgb, i0, i1);
    for (int i = i0; i < i1; ++i) {
      if (!mbar_wait(&full[s], ph, abort)) {
        set_abort(abort, p.status);
        return;
      }
      tc_fence_after();
      const uint32_t a0 = smem_u32(stages + s * SBYTES);
      const uint32_t b0 = a0 + ABYTES;
      // four instructions per stage, each over the next 32 bytes of K
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if constexpr (F8)
          tc_mma_e4m3(d, smem_desc_sw128(a0 + k * 32), smem_desc_sw128(b0 + k * 32), idesc, accumulate);
        else
          tc_mma_bf16(d, smem_desc_sw128(a0 + k * 32), smem_desc_sw128(b0 + k * 32), idesc, accumulate);
        accumulate = 1;
      }
      tc_commit(&empty[s]);
      if (++s == NST) {
        s = 0;
        ph ^= 1;
      }
    }
    tc_commit(&tfull[acc]);
    ++it;
  }
}

// ------------------------------------------------------------------ epilogues
SVL_DEVINL void store_bf16(__nv_bfloat16* dst, const float* v, int n /*16 or 32*/) {
  uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i * 8 < n)
      d[i] = make_uint4(pack_bf16x2(v[8 * i + 0], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                        pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
  }
}

SVL_DEVINL void load_bf16(const __nv_bfloat16* src, float* v, int n) {
  const uint4* s = reinterpret_cast<const uint4*>(src);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i * 8 < n) {
      uint4 u = s[i];
      float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y), c = unpack_bf16x2(u.z), d = unpack_bf16x2(u.w);
      v[8 * i + 0] = a.x; v[8 * i + 1] = a.y; v[8 * i + 2] = b.x; v[8 * i + 3] = b.y;
      v[8 * i + 4] = c.x; v[8 * i + 5] = c.y; v[8 * i + 6] = d.x; v[8 * i + 7] = d.y;
    }
  }
}

// 1 / rms of this row of the residual stream, from its partial sums of squares
SVL_DEVINL float row_rms_scale(const GemmParams& p, int row) {
  float s = 0.f;
  for (int i = 0; i < p.ss_slots; ++i) s += p.ss_in[static_cast<size_t>(i) * p.ss_ld + row];
  return rsqrtf(s * p.ss_inv_d + p.ss_eps);
}

// store_bf16 that also returns the sum of squares of the rounded values
SVL_DEVINL float store_bf16_ss(__nv_bfloat16* dst, const float* v, int n /*16 or 32*/) {
  uint4* d = reinterpret_cast<uint4*>(dst);
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i * 8 < n) {
      uint32_t w[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        w[q] = pack_bf16x2(v[8 * i + 2 * q], v[8 * i + 2 * q + 1]);
        const float2 f = unpack_bf16x2(w[q]);
        ss = fmaf(f.x, f.x, fmaf(f.y, f.y, ss));
      }
      d[i] = make_uint4(w[0], w[1], w[2], w[3]);
    }
  }
  return ss;
}

// e4m3 dequantisation of 32 accumulator columns: v[j] *= f * cs[j] (cs
// 16-byte aligned; the same addresses in every lane of the warp)
SVL_DEVINL void scale_cols(float* v, const float* cs, float f) {
  const float4* c4 = reinterpret_cast<const float4*>(cs);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 c = __ldg(c4 + i);
    v[4 * i] *= f * c.x;
    v[4 * i + 1] *= f * c.y;
    v[4 * i + 2] *= f * c.z;
    v[4 * i + 3] *= f * c.w;
  }
}

template <int KIND, bool F8>
SVL_DEVINL void epilogue_tile(const GemmParams& p, const TileInfo& ti, int row, bool rv,
                              uint32_t taddr) {
  float v[32];
  // row factor of e4m3 operands (the activation row's scale)
  const float af = (F8 && rv) ? p.a_scale[row] : 1.f;
  if constexpr (KIND == EPI_QKV_ROPE) {
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(p.out[ti.mat]);
    const size_t ld = static_cast<size_t>(p.ld[ti.mat]);
    const float rs = ((p.ss_in && rv) ? row_rms_scale(p, row) : 1.f) * af;
    const float* bsc = F8 ? p.b_scale[ti.mat] + ti.n0 : nullptr;
    if (ti.mat < 2) {
      const int dh = p.d_head, half = dh / 2;
      int prow = rv ? p.pos[row] : 0;
      if (prow < 0 || prow >= p.rope_rows) {  // longer than the model's max_seq
        report(p.status, SVL_DEV_BAD_INDEX);
        prow = 0;
      }
      const float2* cs = p.rope_cs + prow;  // frequency i at cs[i * rope_rows]
      float w[32];
      for (int hb = 0; hb < ti.ncols; hb += dh) {
        for (int i0 = 0; i0 < half; i0 += 32) {
          tmem_ld32(taddr + hb + i0, v);
          tmem_ld32(taddr + hb + half + i0, w);
          if (rv) {
            if constexpr (F8) {
              scale_cols(v, bsc + hb + i0, 1.f);
              scale_cols(w, bsc + hb + half + i0, 1.f);
            }
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              const float2 c = cs[static_cast<size_t>(i0 + j) * p.rope_rows];
              const float x1 = v[j] * rs, x2 = w[j] * rs;
              v[j] = x1 * c.x - x2 * c.y;
              w[j] = x2 * c.x + x1 * c.y;
            }
            __nv_bfloat16* o = out + static_cast<size_t>(row) * ld + ti.n0 + hb + i0;
            store_bf16(o, v, 32);
            store_bf16(o + half, w, 32);
          }
        }
      }
    } else {
      // V is stored transposed, V^T[column][row], so that attention reads
      // keys contiguously (ld = padded row count)
      for (int c = 0; c < ti.ncols; c += 32) {
        tmem_ld32(taddr + c, v);
        if (rv) {
          if constexpr (F8) scale_cols(v, bsc + c, 1.f);
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (c + j < ti.ncols) out[static_cast<size_t>(ti.n0 + c + j) * ld + row] = __float2bfloat16_rn(v[j] * rs);
        }
      }
    }
  } else if constexpr (KIND == EPI_RESID) {
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(p.out[0]);
    const size_t ld = static_cast<size_t>(p.ld[0]);
    __nv_bfloat16* orow = out + static_cast<size_t>(row) * ld + ti.n0;
    // residual chunks double-buffered in registers: the load of chunk c+32
    // is in flight while chunk c is added and stored
    uint4 xa[4], xb[4];
    float hss = 0.f;
    if (rv) {
      const uint4* s0 = reinterpret_cast<const uint4*>(orow);
#pragma unroll
      for (int i = 0; i < 4; ++i) xa[i] = (i * 8 < ti.ncols) ? s0[i] : make_uint4(0, 0, 0, 0);
    }
    for (int c = 0; c < ti.ncols; c += 32) {
      const int n = min(32, ti.ncols - c);
      if (rv && c + 32 < ti.ncols) {
        const uint4* s1 = reinterpret_cast<const uint4*>(orow + c + 32);
#pragma unroll
        for (int i = 0; i < 4; ++i) xb[i] = (c + 32 + i * 8 < ti.ncols) ? s1[i] : make_uint4(0, 0, 0, 0);
      }
      tmem_ld32(taddr + c, v);
      if (rv) {
        if constexpr (F8) scale_cols(v, p.b_scale[0] + ti.n0 + c, af);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t w[4] = {xa[i].x, xa[i].y, xa[i].z, xa[i].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 f = unpack_bf16x2(w[q]);
            v[8 * i + 2 * q] += f.x;
            v[8 * i + 2 * q + 1] += f.y;
          }
        }
        if (p.ss_out) {
          hss += store_bf16_ss(orow + c, v, n);
          // one partial per 128 columns of the residual stream
          if (((c + 32) & 127) == 0 || c + 32 >= ti.ncols) {
            p.ss_out[static_cast<size_t>((ti.n0 + c) >> 7) * p.ss_ld + row] = hss;
            hss = 0.f;
          }
        } else {
          store_bf16(orow + c, v, n);
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) xa[i] = xb[i];
    }
  } else if constexpr (KIND == EPI_SWIGLU) {
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(p.out[0]);
    const size_t ld = static_cast<size_t>(p.ld[0]);
    float u[32];
    const float rs = ((p.ss_in && rv) ? row_rms_scale(p, row) : 1.f) * af;
    for (int c = 0; c < ti.ncols; c += 32) {
      tmem_ld32(taddr + c, v);
      tmem_ld32(taddr + kBHalf + c, u);
      if (rv) {
        if constexpr (F8) {
          scale_cols(v, p.b_scale[0] + ti.n0 + c, 1.f);
          scale_cols(u, p.b_scale[1] + ti.n0 + c, 1.f);
        }
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = silu_f(v[j] * rs) * (u[j] * rs);
        store_bf16(out + static_cast<size_t>(row) * ld + ti.n0 + c, v, min(32, ti.ncols - c));
      }
    }
  } else if constexpr (KIND == EPI_GELU || KIND == EPI_ROWMAP) {
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(p.out[0]);
    const size_t ld = static_cast<size_t>(p.ld[0]);
    const int orow = (KIND == EPI_ROWMAP && rv) ? p.row_map[row] : row;
    for (int c = 0; c < ti.ncols; c += 32) {
      tmem_ld32(taddr + c, v);
      if (rv) {
        if constexpr (KIND == EPI_GELU) {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = gelu_f(v[j]);
        }
        store_bf16(out + static_cast<size_t>(orow) * ld + ti.n0 + c, v, min(32, ti.ncols - c));
      }
    }
  } else if constexpr (KIND == EPI_LOGITS_T) {
    float* out = reinterpret_cast<float*>(p.out[0]);
    const size_t ld = static_cast<size_t>(p.ld[0]);
    for (int c = 0; c < ti.ncols; c += 32) {
      tmem_ld32(taddr + c, v);
      if (rv) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (c + j < ti.ncols) out[static_cast<size_t>(ti.n0 + c + j) * ld + row] = v[j];
      }
    }
  } else if constexpr (KIND == EPI_F32) {
    float* out = reinterpret_cast<float*>(p.out[0]);
    const size_t ld = static_cast<size_t>(p.ld[0]);
    for (int c = 0; c < ti.ncols; c += 32) {
      tmem_ld32(taddr + c, v);
      if (rv) {
        if constexpr (F8) scale_cols(v, p.b_scale[0] + ti.n0 + c, af);
        float* o = out + static_cast<size_t>(row) * ld + ti.n0 + c;
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (c + j < ti.ncols) o[j] = v[j];
      }
    }
  } else if constexpr (KIND == EPI_SCORE || KIND == EPI_SCORE_WIDE) {
    // sample of this row: lane 0 searches for the warp's first row, then each
    // lane walks forward (32 consecutive tokens span few samples)
    const int lane = threadIdx.x & 31;
    const int r_first = row - lane;
    int b0 = 0;
    if (lane == 0) {
      int lo = 0, hi = p.n_seg;  // seg_off[lo] <= r_first < seg_off[lo + 1]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (p.seg_off[mid] <= r_first) lo = mid; else hi = mid;
      }
      b0 = lo;
    }
    int b = __shfl_sync(0xffffffffu, b0, 0);
    if (rv)
      while (b + 1 < p.n_seg && p.seg_off[b + 1] <= row) ++b;
    const int H = ti.ncols;
    const float4* eb = reinterpret_cast<const float4*>(p.e_b + static_cast<size_t>(b) * H);
    const uint4* w2v = reinterpret_cast<const uint4*>(p.w2);
    float z = 0.f;
    for (int c = 0; c < H; c += 32) {
      tmem_ld32(taddr + c, v);
      // 32 hidden units: e_b as 8 float4, w2 as 4 x 8 bf16 (H is a multiple of 16)
      const int n = min(32, H - c);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (q * 8 >= n) break;
        const uint4 wq = w2v[(c >> 3) + q];
        const float4 e0 = eb[(c >> 2) + 2 * q], e1 = eb[(c >> 2) + 2 * q + 1];
        const float2 w0 = unpack_bf16x2(wq.x), w1 = unpack_bf16x2(wq.y), w2_ = unpack_bf16x2(wq.z),
                     w3 = unpack_bf16x2(wq.w);
        const int j = 8 * q;
        z += w0.x * silu_f(v[j] + e0.x) + w0.y * silu_f(v[j + 1] + e0.y);
        z += w1.x * silu_f(v[j + 2] + e0.z) + w1.y * silu_f(v[j + 3] + e0.w);
        z += w2_.x * silu_f(v[j + 4] + e1.x) + w2_.y * silu_f(v[j + 5] + e1.y);
        z += w3.x * silu_f(v[j + 6] + e1.z) + w3.y * silu_f(v[j + 7] + e1.w);
      }
    }
    if (rv) {
      z += p.c2;
      if (!isfinite(z)) report(p.status, SVL_DEV_NONFINITE);
      reinterpret_cast<float*>(p.out[0])[row] = z;
    }
  }
}

// Rendezvous of the four epilogue warps around a K-split ticket.
struct KsSync {
  uint64_t* gather;  // 128 arrivals: every row of this share is stored
  uint64_t* done;    // 1 arrival: every share of the tile is stored (*flag = 1) or a wait gave up (0)
  volatile int* flag;
  uint32_t phase;
};

SVL_DEVINL int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Residual epilogue of one K-split share. The share's accumulator goes to
// ks_part; once every share of the tile is stored (the shares run side by
// side in the last wave of the persistent grid, whose CTAs are all resident),
// this CTA sums all shares in order for its 1/nsplit of the tile's rows, adds
// them to the residual rows and writes their norm partial sums. Every wait is
// bounded; returns false on a time-out.
template <bool F8>
SVL_DEVINL bool ksplit_tile(const GemmParams& p, const TileInfo& ti, int lrow, uint32_t taddr, bool empty, KsSync& ks,
                            volatile int* abort) {
  const size_t unit = static_cast<size_t>(ti.slot) * ti.nsplit;
  float* mine = p.ks_part + ((unit + ti.part) * kBM + lrow) * kAccCols;
  // rows past the tile's end are never reduced: no partial for them
  const bool stored = ti.m0 + lrow < ti.m_end;
  float v[32];
  for (int c = 0; c < ti.ncols; c += 32) {
    if (!empty) {
      tmem_ld32(taddr + c, v);  // warp-collective: every lane loads
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = 0.f;
    }
    if (stored) {
      float4* d = reinterpret_cast<float4*>(mine + c);
#pragma unroll
      for (int i = 0; i < 8; ++i) d[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    }
  }
  __threadfence();
  mbar_arrive(ks.gather);
  if (threadIdx.x == 2 * 32) {
    int all = 0;
    if (mbar_wait(ks.gather, ks.phase, abort)) {
      int* ticket = p.ks_ticket + ti.slot;
      atomicAdd(ticket, 1);
      const long long t0 = clock64();
      while (true) {
        if (ld_acquire(ticket) >= ti.nsplit) {
          all = 1;
          break;
        }
        if (*abort || clock64() - t0 > kWaitCycles) break;
      }
    }
    *ks.flag = all;
    mbar_arrive(ks.done);
  }
  const bool got = mbar_wait(ks.done, ks.phase, abort);
  ks.phase ^= 1;
  __syncwarp();
  if (!__all_sync(0xffffffffu, got) || !*ks.flag) return false;
  // The tile's valid rows x 128-column slots form the groups of the
  // reduction; the shares take every nsplit-th group, so the work is spread
  // over all of them even when only a few rows are valid (one row per
  // sample in decode). Four adjacent lanes take the four 32-column chunks of
  // a group and combine their sums of squares for the norm slot.
  const int nr = ti.m_end - ti.m0;
  const int nsl = (ti.ncols + 127) / 128;
  const int ngroups = nr * nsl;
  const int n_mine = ti.part < ngroups ? (ngroups - ti.part + ti.nsplit - 1) / ti.nsplit : 0;
  const int et = threadIdx.x - 2 * 32;  // 0..127
  const int chunk = et & 3;
  const float* base = p.ks_part + unit * kBM * kAccCols;
  for (int k0 = 0; k0 < n_mine; k0 += 32) {  // uniform over the CTA
    const int i = k0 + (et >> 2);
    const bool act = i < n_mine;
    const int g = ti.part + i * ti.nsplit;
    const int lr = act ? g / nsl : 0, sl = act ? g - lr * nsl : 0;
    const int row = ti.m0 + lr;
    const int c = sl * 128 + chunk * 32;
    float hss = 0.f;
    if (act && c < ti.ncols) {
      const int n = min(32, ti.ncols - c);
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = 0.f;
      for (int q = 0; q < ti.nsplit; ++q) {
        const float4* src = reinterpret_cast<const float4*>(base + (static_cast<size_t>(q) * kBM + lr) * kAccCols + c);
        float4 f[8];
#pragma unroll
        for (int i4 = 0; i4 < 8; ++i4) f[i4] = __ldcg(src + i4);
#pragma unroll
        for (int i4 = 0; i4 < 8; ++i4) {
          v[4 * i4] += f[i4].x;
          v[4 * i4 + 1] += f[i4].y;
          v[4 * i4 + 2] += f[i4].z;
          v[4 * i4 + 3] += f[i4].w;
        }
      }
      if constexpr (F8) scale_cols(v, p.b_scale[0] + ti.n0 + c, p.a_scale[row]);
      __nv_bfloat16* orow = reinterpret_cast<__nv_bfloat16*>(p.out[0]) + static_cast<size_t>(row) * p.ld[0] + ti.n0;
      const uint4* xs = reinterpret_cast<const uint4*>(orow + c);
#pragma unroll
      for (int i4 = 0; i4 < 4; ++i4) {
        if (i4 * 8 < n) {
          const uint4 x = xs[i4];
          const uint32_t wd[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float2 f = unpack_bf16x2(wd[k]);
            v[8 * i4 + 2 * k] += f.x;
            v[8 * i4 + 2 * k + 1] += f.y;
          }
        }
      }
      if (p.ss_out) hss = store_bf16_ss(orow + c, v, n);
      else store_bf16(orow + c, v, n);
    }
    if (p.ss_out) {
      // the group's four chunks sit in four adjacent lanes: chunk order kept
      hss += __shfl_xor_sync(0xffffffffu, hss, 1);
      hss += __shfl_xor_sync(0xffffffffu, hss, 2);
      if (act && chunk == 0) p.ss_out[static_cast<size_t>((ti.n0 >> 7) + sl) * p.ss_ld + row] = hss;
    }
  }
  return true;
}

// EPI_RESID through shared memory, for a warp whose 32 rows of the tile all
// exist: 64 columns at a time, the chunk of X that TMA brought into one of
// the warp's two buffers gets the accumulator added in place (bf16, with the
// row's sums of squares of the rounded values for the next norm), and a TMA
// store writes it back. The first two chunks were requested before the
// accumulator was ready; chunk h + 2 is requested once the store of chunk h
// has read its buffer. Bit b of `rpar` is the parity of buffer b's next wait.
template <bool F8>
SVL_DEVINL bool resid_tile_tma(const GemmParams& p, const TileInfo& ti, int q, uint32_t taddr, uint8_t* wst,
                               uint64_t* wbar, uint32_t& rpar, volatile int* abort) {
  const int lane = threadIdx.x & 31;
  const int row = ti.m0 + q * 32 + lane;
  const int nch = ti.ncols / 64;
  const float af = F8 ? p.a_scale[row] : 1.f;
  float hss = 0.f;
  for (int h = 0; h < nch; ++h) {
    const int b = h & 1;
    const bool got = mbar_wait(&wbar[b], (rpar >> b) & 1, abort);
    rpar ^= 1u << b;
    __syncwarp();
    if (!__all_sync(0xffffffffu, got)) return false;
    float v[32], w[32];
    tmem_ld32(taddr + 64 * h, v);
    tmem_ld32(taddr + 64 * h + 32, w);
    if constexpr (F8) {
      scale_cols(v, p.b_scale[0] + ti.n0 + 64 * h, af);
      scale_cols(w, p.b_scale[0] + ti.n0 + 64 * h + 32, af);
    }
    uint8_t* prow = wst + b * kResidChunk + lane * 128;
    float ss[2] = {0.f, 0.f};
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      // 16-byte chunk c of the row, where the 128-byte swizzle put it
      uint4* slot = reinterpret_cast<uint4*>(prow + ((c ^ (lane & 7)) << 4));
      const uint4 x = *slot;
      const float* a = c < 4 ? v + 8 * c : w + 8 * (c - 4);
      const uint32_t xw[4] = {x.x, x.y, x.z, x.w};
      uint32_t o[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float2 f = unpack_bf16x2(xw[k]);
        o[k] = pack_bf16x2(a[2 * k] + f.x, a[2 * k + 1] + f.y);
        const float2 g = unpack_bf16x2(o[k]);
        ss[c >> 2] = fmaf(g.x, g.x, fmaf(g.y, g.y, ss[c >> 2]));
      }
      *slot = make_uint4(o[0], o[1], o[2], o[3]);
    }
    if (p.ss_out) {
      // one partial per 128 columns of the residual stream, its 32-column
      // sums added in column order
      hss += ss[0];
      hss += ss[1];
      if (((64 * h + 64) & 127) == 0 || h + 1 == nch) {
        p.ss_out[static_cast<size_t>((ti.n0 + 64 * h) >> 7) * p.ss_ld + row] = hss;
        hss = 0.f;
      }
    }
    fence_proxy_async();  // generic-proxy writes, read by the TMA unit
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(&p.mapR, wst + b * kResidChunk, ti.n0 + 64 * h, ti.m0 + q * 32);
      bulk_commit();
      if (h + 2 < nch) {
        bulk_wait_read0();  // the store just issued has read this buffer
        mbar_arrive_expect_tx(&wbar[b], kResidChunk);
        tma_load_2d(wst + b * kResidChunk, &p.mapR, &wbar[b], ti.n0 + 64 * (h + 2), ti.m0 + q * 32);
      }
    }
  }
  return true;
}

// EPI_SWIGLU through shared memory, for a warp whose 32 rows of the tile all
// exist: 64 output columns at a time, SiLU(gate) * up goes into one of the
// warp's two buffers (swizzled like the TMA box) and a TMA store writes it
// out. The buffers alternate over all of the warp's chunks (`sbuf` counts
// them), so a buffer is written again once the store before the latest one
// -- its own previous store -- has read it.
template <bool F8>
SVL_DEVINL void swiglu_tile_tma(const GemmParams& p, const TileInfo& ti, int q, uint32_t taddr, uint8_t* wst,
                                uint32_t& sbuf) {
  const int lane = threadIdx.x & 31;
  const int row = ti.m0 + q * 32 + lane;
  const float af = F8 ? p.a_scale[row] : 1.f;
  const float rs = (p.ss_in ? row_rms_scale(p, row) : 1.f) * af;
  const int nch = ti.ncols / 64;
  for (int h = 0; h < nch; ++h) {
    const int b = sbuf++ & 1;
    if (lane == 0) bulk_wait_read1();  // the store before the latest one (from this buffer) has read it
    __syncwarp();
    uint8_t* prow = wst + b * kResidChunk + lane * 128;
#pragma unroll 1
    for (int c2 = 0; c2 < 2; ++c2) {
      float v[32], u[32];
      tmem_ld32(taddr + 64 * h + 32 * c2, v);
      tmem_ld32(taddr + kBHalf + 64 * h + 32 * c2, u);
      if constexpr (F8) {
        scale_cols(v, p.b_scale[0] + ti.n0 + 64 * h + 32 * c2, 1.f);
        scale_cols(u, p.b_scale[1] + ti.n0 + 64 * h + 32 * c2, 1.f);
      }
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = silu_f(v[j] * rs) * (u[j] * rs);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int c = 4 * c2 + i;  // 16-byte chunk of the 128-byte row
        *reinterpret_cast<uint4*>(prow + ((c ^ (lane & 7)) << 4)) =
            make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                       pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
      }
    }
    fence_proxy_async();  // generic-proxy writes, read by the TMA unit
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(&p.mapR, wst + b * kResidChunk, ti.n0 + 64 * h, ti.m0 + q * 32);
      bulk_commit();
    }
  }
}

// 32 bf16 values of this lane's row at column c (a multiple of 32) of the
// warp's staging buffers: buffer c / 64, swizzled like the TMA box.
SVL_DEVINL void stage_row32(uint8_t* wst, int c, const float* v) {
  const int lane = threadIdx.x & 31;
  uint8_t* prow = wst + (c >> 6) * kResidChunk + lane * 128;
  const int pos0 = (c & 63) >> 3;
#pragma unroll
  for (int i = 0; i < 4; ++i)
    *reinterpret_cast<uint4*>(prow + (((pos0 + i) ^ (lane & 7)) << 4)) =
        make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                   pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
}

// EPI_QKV_ROPE, Q and K, through shared memory, for a warp whose 32 rows of
// the tile all exist and heads of a multiple of 64 columns: per head, the
// rotated rows go into the warp's buffers (head columns [0, 64) in the
// first, [64, 128) in the second) and one TMA store per 64 columns writes
// them, once the previous head's stores have read the buffers.
template <bool F8>
SVL_DEVINL void qkv_tile_tma(const GemmParams& p, const TileInfo& ti, int q, uint32_t taddr, uint8_t* wst) {
  const int lane = threadIdx.x & 31;
  const int row = ti.m0 + q * 32 + lane;
  const float af = F8 ? p.a_scale[row] : 1.f;
  const float rs = (p.ss_in ? row_rms_scale(p, row) : 1.f) * af;
  const float* bsc = F8 ? p.b_scale[ti.mat] + ti.n0 : nullptr;
  const CUtensorMap* map = ti.mat == 0 ? &p.mapR : &p.mapR2;
  const int dh = p.d_head, half = dh / 2;
  int prow = p.pos[row];
  if (prow < 0 || prow >= p.rope_rows) {  // longer than the model's max_seq
    report(p.status, SVL_DEV_BAD_INDEX);
    prow = 0;
  }
  const float2* cs = p.rope_cs + prow;  // frequency i at cs[i * rope_rows]
  for (int hb = 0; hb < ti.ncols; hb += dh) {
    if (lane == 0) bulk_wait_read0();  // the previous head's stores have read the buffers
    __syncwarp();
#pragma unroll 1
    for (int i0 = 0; i0 < half; i0 += 32) {
      float v[32], w[32];
      tmem_ld32(taddr + hb + i0, v);
      tmem_ld32(taddr + hb + half + i0, w);
      if constexpr (F8) {
        scale_cols(v, bsc + hb + i0, 1.f);
        scale_cols(w, bsc + hb + half + i0, 1.f);
      }
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float2 c = cs[static_cast<size_t>(i0 + j) * p.rope_rows];
        const float x1 = v[j] * rs, x2 = w[j] * rs;
        v[j] = x1 * c.x - x2 * c.y;
        w[j] = x2 * c.x + x1 * c.y;
      }
      stage_row32(wst, i0, v);
      stage_row32(wst, half + i0, w);
    }
    fence_proxy_async();  // generic-proxy writes, read by the TMA unit
    __syncwarp();
    if (lane == 0) {
      for (int k = 0; k < dh / 64; ++k)
        tma_store_2d(map, wst + k * kResidChunk, ti.n0 + hb + 64 * k, ti.m0 + q * 32);
      bulk_commit();
    }
  }
}

template <int KIND, bool F8, bool THIN>
SVL_DEVINL void epilogue_loop(const GemmParams& p, uint64_t* tfull, uint64_t* tempty, uint32_t tmem,
                              volatile int* abort, KsSync& ks, uint8_t* rstage, uint64_t* rbar) {
  const int ntiles = num_tiles(p);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3;  // TMEM lane quarter this warp may access
  // residual (EPI_RESID) or outputs (EPI_SWIGLU, EPI_QKV_ROPE) through shared memory
  constexpr bool kStaged = (KIND == EPI_RESID || KIND == EPI_SWIGLU || KIND == EPI_QKV_ROPE) && !THIN;
  uint8_t* wst = kStaged ? rstage + q * 2 * kResidChunk : nullptr;
  uint64_t* wbar = kStaged ? rbar + 2 * q : nullptr;
  uint32_t rpar = 0;  // EPI_RESID: parity of each buffer's next wait
  uint32_t sbuf = 0;  // EPI_SWIGLU: chunks stored so far (buffer = sbuf & 1)
  int it = 0;
  for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
    TileInfo ti = get_tile(p, t);
    if (!ti.valid) continue;
    const int acc = it & 1;
    const uint32_t aph = (it >> 1) & 1;
    // (TMA boxes of 64 columns at a 16-byte aligned column)
    const bool staged = kStaged && p.stage_tma && ti.nsplit == 1 && (ti.ncols & 63) == 0 && (ti.n0 & 7) == 0 &&
                        ti.m0 + q * 32 + 32 <= ti.m_end;
    if (staged && KIND == EPI_RESID) {
      // the first two chunks of this warp's rows of X, while the main loop runs
      if (lane == 0) {
        bulk_wait_read0();  // the previous tile's stores have read both buffers
        for (int h = 0; h < 2 && 64 * h < ti.ncols; ++h) {
          mbar_arrive_expect_tx(&wbar[h], kResidChunk);
          tma_load_2d(wst + h * kResidChunk, &p.mapR, &wbar[h], ti.n0 + 64 * h, ti.m0 + q * 32);
        }
      }
    } else if constexpr (KIND == EPI_RESID) {
      // pull this row's residual segment toward L2 while the main loop runs
      const int prow = ti.m0 + q * 32 + lane;
      if (prow < ti.m_end) {
        const char* base = reinterpret_cast<const char*>(
            reinterpret_cast<const __nv_bfloat16*>(p.out[0]) + static_cast<size_t>(prow) * p.ld[0] + ti.n0);
        for (int off = 0; off < ti.ncols * 2; off += 128)
          asm volatile("prefetch.global.L2 [%0];" ::"l"(base + off));
      }
    }
    const bool ok = mbar_wait(&tfull[acc], aph, abort);
    __syncwarp();
    if (!__all_sync(0xffffffffu, ok)) {
      set_abort(abort, p.status);
      return;
    }
    tc_fence_after();
    const int row = ti.m0 + q * 32 + lane;
    const bool rv = row < ti.m_end;
    const uint32_t taddr = tmem + acc * kAccCols + (static_cast<uint32_t>(q * 32) << 16);
    if constexpr (KIND == EPI_RESID) {
      if (ti.nsplit > 1) {
        int i0, i1;
        constexpr int BK = F8 ? kBK8 : kBK;
        k_share(ti, p.K / BK, p.kgroup / BK, i0, i1);
        if (!ksplit_tile<F8>(p, ti, q * 32 + lane, taddr, i0 == i1, ks, abort)) {
          set_abort(abort, p.status);
          return;
        }
      } else if (staged) {
        if (!resid_tile_tma<F8>(p, ti, q, taddr, wst, wbar, rpar, abort)) {
          set_abort(abort, p.status);
          return;
        }
      } else {
        epilogue_tile<KIND, F8>(p, ti, row, rv, taddr);
      }
    } else if (KIND == EPI_SWIGLU && staged) {
      swiglu_tile_tma<F8>(p, ti, q, taddr, wst, sbuf);
    } else if (KIND == EPI_QKV_ROPE && staged && ti.mat < 2 && (p.d_head & 63) == 0) {
      qkv_tile_tma<F8>(p, ti, q, taddr, wst);
    } else {
      epilogue_tile<KIND, F8>(p, ti, row, rv, taddr);
    }
    tc_fence_before();
    mbar_arrive(&tempty[acc]);
    ++it;
  }
  if (kStaged && lane == 0) bulk_wait0();  // this warp's staged stores are complete
}

// ------------------------------------------------------------------ kernel
template <int KIND, bool F8, bool THIN>
__global__ void __launch_bounds__(kGemmThreads, 1) gemm_kernel(const __grid_constant__ GemmParams p) {
  constexpr int NST = StageCfg<KIND, THIN>::stages, SBYTES = StageCfg<KIND, THIN>::bytes;
  constexpr int ABYTES = StageCfg<KIND, THIN>::abytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* stages = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(stages + NST * SBYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + NST;
  uint64_t* tfull = bars + 2 * NST;
  uint64_t* tempty = bars + 2 * NST + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * NST + 4);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  KsSync ks{bars + 2 * NST + 5, bars + 2 * NST + 6, reinterpret_cast<volatile int*>(bars + 2 * NST + 7), 0};
  // EPI_RESID / EPI_SWIGLU / EPI_QKV_ROPE: the epilogue warps' chunk buffers
  // (and, for the residual loads, their barriers)
  constexpr bool kStaged = (KIND == EPI_RESID || KIND == EPI_SWIGLU || KIND == EPI_QKV_ROPE) && !THIN;
  uint64_t* rbar = bars + 2 * NST + 8;
  uint8_t* rstage = stages + NST * SBYTES + 1024;
  static_assert(!kStaged || (2 * NST + 16) * 8 <= 256, "barriers of the staged residual epilogue");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < NST; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 4 * 32);
    }
    mbar_init(ks.gather, 4 * 32);
    mbar_init(ks.done, 1);
    if (kStaged)
      for (int i = 0; i < 8; ++i) mbar_init(&rbar[i], 1);
    *abort = 0;
    fence_barrier_init();
    fence_proxy_async();
    prefetch_tmap(&p.mapA);
    prefetch_tmap(&p.mapB[0]);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // set-up above touches no global data; from here on the predecessor's
  // outputs are read
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) producer_loop<NST, SBYTES, ABYTES, F8>(p, stages, full, empty, abort);
  } else if (warp == 1) {
    if (lane == 0) mma_loop<NST, SBYTES, ABYTES, F8>(p, stages, full, empty, tfull, tempty, tmem, abort);
  } else {
    epilogue_loop<KIND, F8, THIN>(p, tfull, tempty, tmem, abort, ks, rstage, rbar);
  }

  __syncwarp();
  if (*abort) {
    // Let copies and MMAs already issued land before the CTA lets go of its
    // shared and tensor memory (about 10 ms; they finish in microseconds).
    long long t0 = clock64();
    while (clock64() - t0 < 20000000LL) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ CTA-pair kernel
// The same GEMM on 256-row tiles computed by a cluster of two CTAs on two SMs
// (tcgen05 cta_group::2). Each CTA loads its 128 rows of A and half of B (the
// first or the second N/2 rows of the tile's B, or the gate or the up rows of
// a gate/up tile) into its own shared memory; the leader (cluster rank 0)
// issues the MMAs, which read both CTAs' halves and write D rows 0-127 into
// the leader's tensor memory and rows 128-255 into the peer's. Per SM and K
// block this moves 32 KB through shared memory for a 128 x N product where the
// single-CTA kernel moves 48 KB, which is what caps that kernel's tensor pipe.
//
//   full[s]    leader only: both CTAs' TMA loads of stage s (the leader posts
//              the byte count of both, the peer's loads complete on it);
//   empty[s]   each CTA: stage s consumed (the leader's MMA commit, multicast);
//   tfull[a]   each CTA: accumulator a ready (commit, multicast);
//   tempty[a]  leader only: both CTAs' epilogues have read accumulator a.
// Waits are bounded as in the single-CTA kernel. The two cluster barriers (after
// set-up and before the tensor memory is released) are reached by every thread
// of both CTAs on every path; each producer first waits for the release of its
// last stages, so no MMA completion can arrive after its CTA has exited.
#ifndef SVL_PAIR_STAGES
#define SVL_PAIR_STAGES 6
#endif
constexpr int kPairStages = SVL_PAIR_STAGES;
constexpr int kPairBox = 64;                         // B rows per TMA box (64-row tensor maps)
constexpr int kPairBBytes = kBHalf * kBK * 2;        // up to 128 B rows per CTA
constexpr int kPairStageBytes = kABytes + kPairBBytes;
constexpr int kPairSmem = kPairStages * kPairStageBytes + 1024 + 256;
static_assert(kPairSmem <= 232448, "shared memory per CTA");

// MMA N of a pair tile: gate/up tiles are 128 gate + 128 up rows; others
// round their columns up to 128 or 256 (each CTA holds N / 2 rows of B).
SVL_DEVINL int pair_n(const GemmParams& p, const TileInfo& ti) {
  if (p.b_split) return 2 * kBHalf;
  return ti.ncols > kBHalf ? 2 * kBHalf : kBHalf;
}

SVL_DEVINL void pair_producer(const GemmParams& p, uint8_t* stages, uint64_t* full, uint64_t* empty, uint32_t rank,
                              volatile int* abort) {
  const int ntiles = num_tiles(p);
  const int npairs = gridDim.x >> 1, pair = blockIdx.x >> 1;
  const int nkb = p.K / kBK, kgb = p.kgroup / kBK;
  int s = 0;
  uint32_t ph = 0;
  auto next = [&]() {
    if (++s == kPairStages) {
      s = 0;
      ph ^= 1;
    }
  };
  for (int t = pair; t < ntiles; t += npairs) {
    const TileInfo ti = get_tile(p, t);
    if (!ti.valid) continue;
    const int brows = pair_n(p, ti) / 2;
    const CUtensorMap* mb = p.b_split ? &p.mapB[rank] : &p.mapB[ti.mat];
    const int by = p.b_split ? ti.n0 : ti.n0 + static_cast<int>(rank) * brows;
    const uint32_t bytes = 2u * static_cast<uint32_t>(kABytes + brows * 128);
    KWalk w(nkb, kgb, ti.kmask);
    while (w.next()) {
      if (!mbar_wait(&empty[s], ph ^ 1, abort)) {
        set_abort(abort, p.status);
        return;
      }
      uint8_t* sa = stages + s * kPairStageBytes;
      uint8_t* sb = sa + kABytes;
      if (rank == 0) mbar_arrive_expect_tx(&full[s], bytes);
      const uint32_t fb = mapa_shared(&full[s], 0);
      tma_load_2d_pair(sa, &p.mapA, fb, w.kb * kBK, ti.m0 + static_cast<int>(rank) * kBM);
      for (int r = 0; r < brows; r += kPairBox) tma_load_2d_pair(sb + r * 128, mb, fb, w.kb * kBK, by + r);
      next();
    }
  }
  // the releases of the last stages (the leader's MMA commits) have arrived here
  for (int i = 0; i < kPairStages; ++i) {
    if (!mbar_wait(&empty[s], ph ^ 1, abort)) {
      set_abort(abort, p.status);
      return;
    }
    next();
  }
}

SVL_DEVINL void pair_mma(const GemmParams& p, uint8_t* stages, uint64_t* full, uint64_t* empty, uint64_t* tfull,
                         uint64_t* tempty, uint32_t tmem, volatile int* abort) {
  const int ntiles = num_tiles(p);
  const int npairs = gridDim.x >> 1, pair = blockIdx.x >> 1;
  const int nkb = p.K / kBK, kgb = p.kgroup / kBK;
  int s = 0, it = 0;
  uint32_t ph = 0;
  for (int t = pair; t < ntiles; t += npairs) {
    const TileInfo ti = get_tile(p, t);
    if (!ti.valid) continue;
    const int acc = it & 1;
    const uint32_t aph = (it >> 1) & 1;
    if (!mbar_wait(&tempty[acc], aph ^ 1, abort)) {
      set_abort(abort, p.status);
      return;
    }
    tc_fence_after();
    const uint32_t idesc = idesc_bf16_f32(2 * kBM, pair_n(p, ti));
    const uint32_t d = tmem + acc * kAccCols;
    uint32_t accumulate = 0;
    KWalk w(nkb, kgb, ti.kmask);
    while (w.next()) {
      if (!mbar_wait(&full[s], ph, abort)) {
        set_abort(abort, p.status);
        return;
      }
      tc_fence_after();
      const uint32_t a0 = smem_u32(stages + s * kPairStageBytes);
      const uint32_t b0 = a0 + kABytes;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        tc_mma_bf16_pair(d, smem_desc_sw128(a0 + k * 32), smem_desc_sw128(b0 + k * 32), idesc, accumulate);
        accumulate = 1;
      }
      tc_commit_pair(&empty[s]);
      if (++s == kPairStages) {
        s = 0;
        ph ^= 1;
      }
    }
    tc_commit_pair(&tfull[acc]);
    ++it;
  }
}

template <int KIND>
SVL_DEVINL void pair_epilogue(const GemmParams& p, uint64_t* tfull, uint64_t* tempty, uint32_t tmem, uint32_t rank,
                              volatile int* abort) {
  const int ntiles = num_tiles(p);
  const int npairs = gridDim.x >> 1, pair = blockIdx.x >> 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3;  // TMEM lane quarter this warp may access
  int it = 0;
  for (int t = pair; t < ntiles; t += npairs) {
    const TileInfo ti = get_tile(p, t);
    if (!ti.valid) continue;
    const int acc = it & 1;
    const uint32_t aph = (it >> 1) & 1;
    const bool ok = mbar_wait(&tfull[acc], aph, abort);
    __syncwarp();
    if (!__all_sync(0xffffffffu, ok)) {
      set_abort(abort, p.status);
      return;
    }
    tc_fence_after();
    const int row = ti.m0 + static_cast<int>(rank) * kBM + q * 32 + lane;
    const uint32_t taddr = tmem + acc * kAccCols + (static_cast<uint32_t>(q * 32) << 16);
    epilogue_tile<KIND, false>(p, ti, row, row < ti.m_end, taddr);
    tc_fence_before();
    if (rank == 0)
      mbar_arrive(&tempty[acc]);
    else
      mbar_arrive_cluster(mapa_shared(&tempty[acc], 0));
    ++it;
  }
}

template <int KIND>
__global__ void __launch_bounds__(kGemmThreads, 1) gemm_pair_kernel(const __grid_constant__ GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* stages = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(stages + kPairStages * kPairStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kPairStages;
  uint64_t* tfull = bars + 2 * kPairStages;
  uint64_t* tempty = bars + 2 * kPairStages + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kPairStages + 4);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t rank = cluster_rank();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kPairStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 2 * 4 * 32);  // the epilogue threads of both CTAs
    }
    *abort = 0;
    fence_barrier_init();
    fence_proxy_async();
    prefetch_tmap(&p.mapA);
    prefetch_tmap(&p.mapB[0]);
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_sync();  // both CTAs' barriers exist before any TMA or arrive reaches them
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) pair_producer(p, stages, full, empty, rank, abort);
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) pair_mma(p, stages, full, empty, tfull, tempty, tmem, abort);
  } else {
    pair_epilogue<KIND>(p, tfull, tempty, tmem, rank, abort);
  }

  __syncwarp();
  if (*abort) {
    // let copies and MMAs already issued land before shared and tensor memory go
    long long t0 = clock64();
    while (clock64() - t0 < 20000000LL) {
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the peer is done with this CTA's barriers and tensor memory
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
}

template <int KIND>
static cudaError_t launch_pair_kind(const GemmParams& p, int pairs, cudaStream_t stream) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(gemm_pair_kernel<KIND>, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(2 * pairs));
  cfg.blockDim = dim3(kGemmThreads);
  cfg.dynamicSmemBytes = kPairSmem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, gemm_pair_kernel<KIND>, p);
}

cudaError_t launch_gemm_pair(EpiKind kind, const GemmParams& p, int pairs, cudaStream_t stream) {
  if (pairs <= 0) return cudaSuccess;
  switch (kind) {
    case EPI_QKV_ROPE: return launch_pair_kind<EPI_QKV_ROPE>(p, pairs, stream);
    case EPI_SWIGLU: return launch_pair_kind<EPI_SWIGLU>(p, pairs, stream);
    default: return cudaErrorInvalidValue;
  }
}

int gemm_pair_max_clusters(EpiKind kind) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(kGemmThreads);
  cfg.dynamicSmemBytes = kPairSmem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  cudaError_t e;
  if (kind == EPI_QKV_ROPE) {
    e = cudaFuncSetAttribute(gemm_pair_kernel<EPI_QKV_ROPE>, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, gemm_pair_kernel<EPI_QKV_ROPE>, &cfg);
  } else {
    e = cudaFuncSetAttribute(gemm_pair_kernel<EPI_SWIGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, gemm_pair_kernel<EPI_SWIGLU>, &cfg);
  }
  return e == cudaSuccess ? n : 0;
}

// Dynamic shared memory of gemm_kernel: the stages, the alignment slack and
// the barriers, and for the staged residual epilogue its chunk buffers (at
// the next 1024-byte boundary after the barriers).
template <int KIND, bool THIN>
constexpr int gemm_smem() {
  return StageCfg<KIND, THIN>::stages * StageCfg<KIND, THIN>::bytes + 1024 + 256 +
         (((KIND == EPI_RESID || KIND == EPI_SWIGLU || KIND == EPI_QKV_ROPE) && !THIN) ? 1024 - 256 + kResidStageBytes
                                                                                      : 0);
}

template <int KIND, bool F8 = false, bool THIN = false>
static cudaError_t launch_kind(const GemmParams& p, int grid, cudaStream_t stream) {
  constexpr int smem = gemm_smem<KIND, THIN>();
  static_assert(smem <= 232448, "shared memory per CTA");
  static bool configured = false;
  if (!configured) {
    cudaError_t e =
        cudaFuncSetAttribute(gemm_kernel<KIND, F8, THIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  return launch_pdl(gemm_kernel<KIND, F8, THIN>, grid, kGemmThreads, smem, stream, p);
}

template <int KIND, bool F8, bool THIN>
static int blocks_per_sm_kind() {
  constexpr int smem = gemm_smem<KIND, THIN>();
  int n = 0;
  if (cudaFuncSetAttribute(gemm_kernel<KIND, F8, THIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
          cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemm_kernel<KIND, F8, THIN>, kGemmThreads, smem) !=
          cudaSuccess)
    return 0;
  return n;
}

int gemm_resid_blocks_per_sm(bool e4m3) {
  const int a = e4m3 ? blocks_per_sm_kind<EPI_RESID, true, false>() : blocks_per_sm_kind<EPI_RESID, false, false>();
  const int b = e4m3 ? blocks_per_sm_kind<EPI_RESID, true, true>() : blocks_per_sm_kind<EPI_RESID, false, true>();
  return a < b ? a : b;
}

cudaError_t launch_gemm(EpiKind kind, const GemmParams& p, int grid, cudaStream_t stream, bool e4m3, bool thin) {
  if (e4m3 && (!p.a_scale || !p.b_scale[0])) return cudaErrorInvalidValue;
  if (thin) {
    switch (kind) {
      case EPI_QKV_ROPE:
        return e4m3 ? launch_kind<EPI_QKV_ROPE, true, true>(p, grid, stream)
                    : launch_kind<EPI_QKV_ROPE, false, true>(p, grid, stream);
      case EPI_RESID:
        return e4m3 ? launch_kind<EPI_RESID, true, true>(p, grid, stream)
                    : launch_kind<EPI_RESID, false, true>(p, grid, stream);
      case EPI_SWIGLU:
        return e4m3 ? launch_kind<EPI_SWIGLU, true, true>(p, grid, stream)
                    : launch_kind<EPI_SWIGLU, false, true>(p, grid, stream);
      default: return cudaErrorInvalidValue;
    }
  }
  if (e4m3) {
    switch (kind) {
      case EPI_QKV_ROPE: return launch_kind<EPI_QKV_ROPE, true>(p, grid, stream);
      case EPI_RESID: return launch_kind<EPI_RESID, true>(p, grid, stream);
      case EPI_SWIGLU: return launch_kind<EPI_SWIGLU, true>(p, grid, stream);
      case EPI_F32: return launch_kind<EPI_F32, true>(p, grid, stream);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (kind) {
    case EPI_QKV_ROPE: return launch_kind<EPI_QKV_ROPE>(p, grid, stream);
    case EPI_RESID: return launch_kind<EPI_RESID>(p, grid, stream);
    case EPI_SWIGLU: return launch_kind<EPI_SWIGLU>(p, grid, stream);
    case EPI_GELU: return launch_kind<EPI_GELU>(p, grid, stream);
    case EPI_ROWMAP: return launch_kind<EPI_ROWMAP>(p, grid, stream);
    case EPI_LOGITS_T: return launch_kind<EPI_LOGITS_T>(p, grid, stream);
    case EPI_F32: return launch_kind<EPI_F32>(p, grid, stream);
    case EPI_SCORE: return launch_kind<EPI_SCORE>(p, grid, stream);
    case EPI_SCORE_WIDE: return launch_kind<EPI_SCORE_WIDE>(p, grid, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace svl
