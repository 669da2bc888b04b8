// Persistent tcgen05/TMEM GEMM for sm_103a: C[M,N] = A[M,K] * B[N,K]^T with
// bf16 (or, for the gated projections, e4m3) K-major operands staged by TMA
// (128-byte swizzle) and an fp32 accumulator in tensor memory, followed by a
// fused epilogue.
//
// Work arrives either as an explicit device tile list (the gated layers: one
// tile per (row segment, column run) of active groups) or as a dense grid.
#pragma once

#include "common.cuh"

namespace svl {

constexpr int kBM = 128;           // rows per tile (TMEM lanes)
constexpr int kBK = 64;            // K per stage: one 128-byte swizzle row (bf16)
constexpr int kBK8 = 128;          // the same 128 bytes of e4m3
constexpr int kBHalf = 128;        // B rows per TMA box; a stage holds two
constexpr int kStages = 4;
constexpr int kThinRows = 32;      // A rows of a THIN launch (see launch_gemm)
constexpr int kABytes = kBM * kBK * 2;
constexpr int kBHalfBytes = kBHalf * kBK * 2;
constexpr int kStageBytes = kABytes + 2 * kBHalfBytes;
constexpr int kGemmThreads = 192;  // warp 0 TMA, warp 1 MMA + TMEM, warps 2-5 epilogue
constexpr int kAccCols = 256;      // fp32 columns per accumulator
constexpr int kTmemCols = 512;     // two accumulators (epilogue overlaps the next tile)
constexpr int kGemmSmem = kStages * kStageBytes + 1024 /*align*/ + 256 /*barriers*/;
constexpr int kResidChunk = 32 * 128;             // one warp's 32 rows x 64 columns of bf16 (staged epilogues)
constexpr int kResidStageBytes = 4 * 2 * kResidChunk;  // two chunk buffers per epilogue warp

enum EpiKind : int {
  EPI_QKV_ROPE = 0,  // mat 0/1: RoPE then bf16 store to Q/K; mat 2: bf16 store to V^T (transposed)
  EPI_RESID = 1,     // out[r, n] = bf16(out[r, n] + acc)
  EPI_SWIGLU = 2,    // out[r, n0 + c] = bf16(SiLU(acc[c]) * acc[128 + c])
  EPI_GELU = 3,      // out[r, n] = bf16(GELU(acc))
  EPI_ROWMAP = 4,    // out[row_map[r], n] = bf16(acc)
  EPI_LOGITS_T = 5,  // out[n, r] = acc (fp32): swapped LM head, r = vocab id, n = sample
  EPI_F32 = 6,       // out[r, n] = acc (fp32)
  EPI_SCORE = 7,     // z[r] = sum_h w2[h] SiLU(acc[h] + e_b[sample(r), h]) + c2, H <= 64
  EPI_SCORE_WIDE = 8,  // the same for 64 < H <= 128 (larger B boxes, fewer stages)
  EPI_COUNT = 8
};

// Tile encoding (int4): x = m0, y = m_end (rows >= m_end are not stored),
// z = n0, w = ncols | mat << 16 | kmask << 24 (kmask 0 = every K block).
SVL_DEVINL int tile_ncols(int w) { return w & 0xFFFF; }
SVL_DEVINL int tile_mat(int w) { return (w >> 16) & 0xFF; }
SVL_DEVINL int tile_kmask(int w) { return (w >> 24) & 0xFF; }

struct GemmParams {
  CUtensorMap mapA;
  CUtensorMap mapB[3];
  // explicit tile list (tiles != nullptr) ...
  const int4* tiles;
  const int* tile_count;
  int max_tiles;
  // ... or dense grid: grid_m x grid_n tiles of kBM x bn
  int grid_m, grid_n, bn;
  const int* m_limit_dev;  // rows bound read on the device (nullptr: use m_limit)
  int m_limit, n_limit;
  // K loop
  int K;       // multiple of 64 (e4m3: 128)
  int kgroup;  // K elements per gate group (kmask), multiple of 64 (e4m3: 128)
  int b_split; // 1: B rows 0-127 from mapB[0], rows 128-255 from mapB[1] (gate | up)
  int b_box_rows;  // rows of one B box when mapB has boxes of fewer than 128 rows (0: 128)
  // epilogue operands
  void* out[3];
  int ld[3];
  const int* row_map;
  const int* pos;
  const float2* rope_cs;  // [d_head/2, rope_rows] (cos, sin), position fastest
  int rope_rows;
  int d_head;
  const float* e_b;       // [B, H]
  const int* seg_off;     // [B+1] token offsets per sample (score)
  int n_seg;
  const __nv_bfloat16* w2;
  float c2;
  // RMSNorm fused into the GEMMs around it: per-row partial sums of squares
  // of the residual stream, one slot per 128 columns ([slot][row], ss_ld
  // floats apart). The residual epilogue writes the slots of the columns it
  // stores (ss_out); the QKV and gate/up epilogues sum a row's ss_slots slots
  // and scale its accumulator by 1/sqrt(sum/D + eps) (ss_in).
  const float* ss_in;
  float* ss_out;
  int ss_ld, ss_slots;
  float ss_inv_d, ss_eps;
  // K-split tail (residual GEMMs): from tile index ks_info[0] on, the list
  // holds the ks_info[1] tail tiles repeated ks_info[2] times; copy `part`
  // of tail tile `slot` computes that share of the tile's active K blocks and
  // stores it to ks_part, counts itself in ks_ticket[slot] and, once all
  // shares are in, reduces its own slice of the tile's rows. Tickets start
  // at zero (a separate array per launch).
  const int* ks_info;  // [3] on the device, or nullptr
  float* ks_part;      // [tail tiles * parts][128][256]
  int* ks_ticket;      // [tail tiles]
  // e4m3 operands (QKV, residual and SwiGLU epilogues): the accumulator is
  // the sum of code products; the epilogue scales element (r, n) by
  // a_scale[r] * b_scale[mat][n] before anything else. The b_scale arrays
  // are readable 32 floats past their last column.
  const float* a_scale;
  const float* b_scale[3];
  // out[0] as a tensor map with boxes of 64 columns x 32 rows (EPI_RESID:
  // the residual stream; EPI_SWIGLU: the hidden rows; EPI_QKV_ROPE: Q, and K
  // in mapR2). When stage_tma is set, each epilogue warp whose 32 rows of a
  // tile all exist stages them through shared memory: EPI_RESID loads X with
  // TMA, adds the accumulator and stores back; EPI_SWIGLU and EPI_QKV_ROPE (Q
  // and K) write their outputs and store them with TMA (per-thread loads and
  // stores otherwise, and for V^T).
  CUtensorMap mapR;
  CUtensorMap mapR2;  // EPI_QKV_ROPE: mapR holds Q (mat 0), mapR2 K (mat 1)
  int stage_tma;
  // 1: A loads with the L2 evict_first policy. The n-band lists of the
  // residual GEMMs keep a band of weights in L2 while the input rows stream
  // through; this keeps the rows from pushing the band out.
  int a_evict_first;
  uint32_t* status;
};

// `thin`: every tile has at most kThinRows rows and mapA has boxes of
// kThinRows rows (QKV, residual and SwiGLU epilogues): deeper weight
// pipeline for decode-sized batches.
cudaError_t launch_gemm(EpiKind kind, const GemmParams& p, int grid, cudaStream_t stream, bool e4m3 = false,
                        bool thin = false);

// The gated QKV / gate-up GEMM on 256-row tiles by clusters of two CTAs
// (tcgen05 cta_group::2): `pairs` clusters walk the tile list (tiles of up to
// 256 rows), mapA has 128-row boxes, mapB 64-row boxes. bf16 only.
cudaError_t launch_gemm_pair(EpiKind kind, const GemmParams& p, int pairs, cudaStream_t stream);
// Clusters of two of the pair kernel that can be resident at once (0 if the
// query fails).
int gemm_pair_max_clusters(EpiKind kind);

// CTAs of the residual (EPI_RESID) GEMM that fit on one SM at once, the
// smaller of the wide and THIN instantiations (0 if the query fails).
int gemm_resid_blocks_per_sm(bool e4m3);

}  // namespace svl
