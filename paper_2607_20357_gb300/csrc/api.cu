// C ABI of the gated prefill: argument checks, model state, workspace layout,
// tensor-map encoding and the launch sequences of the three stages.
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdlib>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "gemm.cuh"
#include "kernels.cuh"

using namespace svl;

struct svl_model {
  svl_model_desc d;
  svl_weights w;
  std::vector<svl_layer_weights> layers;
  int device = 0;
  int num_sms = 0;
  // every CTA of the persistent residual GEMM fits on the GPU at once, so
  // the shares of a K-split tail can wait for each other (else no split)
  bool ks_resident = false;
  // QKV and gate/up on CTA pairs (256-row tiles, tcgen05 cta_group::2):
  // clusters of two resident at once (0: single-CTA kernel); per layer the
  // q, k, v, g, u weights as tensor maps with 64-row boxes
  int pair_clusters = 0;
  std::vector<CUtensorMap> tm_pair;
  uint32_t* d_status = nullptr;
  float2* rope_cs = nullptr;
  // B-operand tensor maps of the weights: per layer q, k, v, o, g, u, d
  std::vector<CUtensorMap> tm_layer;
  // norm gains folded into the projections after them (allocated only for
  // layers whose gains are not all ones): per layer q, k, v, g, u or nullptr
  std::vector<void*> folded;
  CUtensorMap tm_ctrl_w1, tm_proj_w1, tm_proj_w2, tm_lm_head;
  // e4m3 gated projections (gemm_format SVL_GEMM_E4M3): per layer the codes
  // of q, k, v, o, g, u, d with their per-row scales, and uint8 tensor maps.
  // The O and down weights hold each group's K columns padded to a multiple
  // of 128 (one K block), so that gated-off groups skip whole blocks.
  bool e4m3 = false;
  int kgo_p = 0, kgd_p = 0;
  std::vector<void*> f8_mem;           // one allocation per layer
  std::vector<const float*> f8_scale;  // per layer q, k, v, o, g, u, d
  std::vector<CUtensorMap> tm8;        // per layer q, k, v, o, g, u, d
  // kernel timing (svl_profile_start / svl_profile_stop)
  bool prof = false;
  uint32_t prof_mask = 0;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  std::vector<std::pair<int, size_t>> prof_recs;  // (tag, index of the first event of the pair)
  std::vector<std::pair<int, float>> prof_last;   // per-launch times of the last window
};

namespace {

std::atomic<uint64_t> g_launches{0};

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D bf16 tensor map, K-major rows of `cols` elements, boxes of 64 x 128
// with 128-byte swizzle (the layout the tcgen05 descriptors expect).
bool make_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows = 128) {
  auto fn = encode_fn();
  if (!fn || !ptr || rows == 0 || cols == 0 || (reinterpret_cast<uintptr_t>(ptr) & 15) || ((cols * 2) & 15))
    return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The same for uint8 e4m3 codes: boxes of 128 x box_rows (128 bytes per row).
bool make_map8(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows = 128) {
  auto fn = encode_fn();
  if (!fn || !ptr || rows == 0 || cols == 0 || (reinterpret_cast<uintptr_t>(ptr) & 15) || (cols & 15)) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK8), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int round128(int x) { return (x + 127) & ~127; }

constexpr int kMaxPrefillBatch = 4096;  // samples per prefill call

// Each call keeps its scratch at the start of the workspace: no data flows
// between calls through the workspace, so the three layouts overlap and the
// workspace size is the largest of them.
struct SelLayout {
  size_t e_b, scalars, kept_local, total;
};
struct PackLayout {
  size_t scalars, stage, hp, row_map, tok, total;
};
struct PreLayout {
  int64_t t_cap, t_pad;
  int n_pad, mt_max, qkv_cap, o_cap, gu_cap, dn_cap, attn_cap;
  int ss_slots, ks_units;
  int64_t aq_cols;  // e4m3: widest quantised activation row (0 for bf16)
  size_t xn, q, k, v, ao, hmid, yl, ss_a, ss_b, ks_part, ks_ticket, ks_info, act, seg, qkv, o, gu, dn, attn, counts,
      aq, as, total;
};

struct Bump {
  size_t off = 0;
  size_t take(size_t bytes) {
    size_t o = off;
    off = align256(off + bytes);
    return o;
  }
};

SelLayout sel_layout(const svl_model_desc& d, int B, int64_t nv) {
  SelLayout L{};
  Bump b;
  L.e_b = b.take(sizeof(float) * B * d.h_ctrl);
  L.scalars = b.take(64);
  L.kept_local = b.take(sizeof(int) * std::max<int64_t>(nv, 1));
  L.total = b.off;
  return L;
}

PackLayout pack_layout(const svl_model_desc& d, int B, int64_t nv) {
  PackLayout L{};
  Bump b;
  L.scalars = b.take(64);
  L.tok = b.take(2 * static_cast<size_t>(B) * d.d_model);  // budget-token rows (compute controller)
  if (d.proj_hidden) {
    L.stage = b.take(2 * nv * d.c_vis);
    L.hp = b.take(2 * nv * d.proj_hidden);
    L.row_map = b.take(sizeof(int) * std::max<int64_t>(nv, 1));
  }
  L.total = b.off;
  return L;
}

PreLayout pre_layout(const svl_model_desc& d, int B, int64_t t_cap) {
  PreLayout L{};
  const int64_t dh = d.d_model / d.n_heads, dkv = static_cast<int64_t>(d.n_kv_heads) * dh;
  const int64_t hq = static_cast<int64_t>(d.n_heads) * dh;
  const int G = d.n_groups;
  L.t_cap = t_cap;
  L.t_pad = (t_cap + 7) & ~int64_t(7);
  L.n_pad = ((B + 15) / 16) * 16;
  L.mt_max = static_cast<int>(t_cap / 128 + B + 1);
  const int qkv_nt = static_cast<int>((hq / 256 + G + 1) + 2 * (dkv / 256 + G + 1));
  // + 256: room for the split tail (at most half a wave of extra tiles)
  L.qkv_cap = L.mt_max * qkv_nt + 256;
  L.o_cap = L.mt_max * ((d.d_model + 255) / 256) + 256;
  L.dn_cap = L.o_cap;
  L.gu_cap = L.mt_max * (d.d_ffn / 128 + G + 1);
  L.attn_cap = static_cast<int>(d.n_heads * (t_cap / kAttnQ + B + 1));
  Bump b;
  L.xn = b.take(2 * t_cap * d.d_model);
  L.q = b.take(2 * t_cap * hq);
  L.k = b.take(2 * t_cap * dkv);
  L.v = b.take(2 * L.t_pad * dkv);  // V^T [dkv, t_pad]
  L.ao = b.take(2 * t_cap * hq);
  L.hmid = b.take(2 * t_cap * d.d_ffn);
  L.yl = b.take(2 * static_cast<size_t>(L.n_pad) * d.d_model);
  // partial sums of squares of the residual stream, [D/128][t_pad] each: A
  // feeds the attention input norm, B the MLP input norm
  L.ss_slots = d.d_model / 128;
  L.ss_a = b.take(sizeof(float) * L.ss_slots * L.t_pad);
  L.ss_b = b.take(sizeof(float) * L.ss_slots * L.t_pad);
  // K-split tail of the residual GEMMs: at most 8 shares per tail tile and
  // 256 shares in all, fp32 128 x 256 each
  L.ks_units = static_cast<int>(std::min<int64_t>(256, 8LL * L.mt_max * ((d.d_model + 255) / 256)));
  L.ks_part = b.take(sizeof(float) * static_cast<size_t>(L.ks_units) * kBM * 256);
  const size_t nl = d.n_layers;
  L.ks_ticket = b.take(sizeof(int) * L.ks_units * 2 * nl);  // per layer and residual GEMM
  L.ks_info = b.take(sizeof(int) * 8 * nl);
  L.act = b.take(nl * B);
  L.seg = b.take(sizeof(int4) * nl * B);
  L.qkv = b.take(sizeof(int4) * nl * L.qkv_cap);
  L.o = b.take(sizeof(int4) * nl * L.o_cap);
  L.gu = b.take(sizeof(int4) * nl * L.gu_cap);
  L.dn = b.take(sizeof(int4) * nl * L.dn_cap);
  L.attn = b.take(sizeof(int4) * nl * L.attn_cap);
  L.counts = b.take(sizeof(int) * 6 * nl);  // five tile/item counts and the attention unit counters
  // e4m3: the quantised rows of the current GEMM input and their scales
  if (d.gemm_format == SVL_GEMM_E4M3) {
    const int64_t o_cols = static_cast<int64_t>(G) * round128(static_cast<int>(hq / G));
    const int64_t d_cols = static_cast<int64_t>(G) * round128(d.d_ffn / G);
    L.aq_cols = std::max<int64_t>(d.d_model, std::max(o_cols, d_cols));
    L.aq = b.take(static_cast<size_t>(t_cap) * L.aq_cols);
    L.as = b.take(sizeof(float) * (t_cap + 64));
  }
  L.total = b.off;
  return L;
}

// Device copies of the inputs and intermediate outputs of
// svl_prefill_from_host; the stage scratch follows at `inner`.
struct HostLayout {
  size_t vis, vis_off, text_ids, text_off, text_len, budget, keep, lg, gg;
  size_t scores, k, kept_idx, kept_off, flags, X, cu, pos, logits, inner, total;
};

HostLayout host_layout(const svl_model_desc& d, int B, int64_t nv, int64_t nt) {
  HostLayout L{};
  Bump b;
  const int64_t t_cap = std::max<int64_t>(nv + nt, 1);
  L.vis = b.take(2 * std::max<int64_t>(nv, 1) * d.c_vis);
  L.vis_off = b.take(4 * (B + 1));
  L.text_ids = b.take(4 * std::max<int64_t>(nt, 1));
  L.text_off = b.take(4 * (B + 1));
  L.text_len = b.take(4 * B);
  L.budget = b.take(4 * B);
  L.keep = b.take(4 * B);
  L.lg = b.take(static_cast<size_t>(B) * d.n_layers);
  L.gg = b.take(static_cast<size_t>(B) * d.n_layers * d.n_groups);
  L.scores = b.take(4 * std::max<int64_t>(nv, 1));
  L.k = b.take(4 * B);
  L.kept_idx = b.take(4 * std::max<int64_t>(nv, 1));
  L.kept_off = b.take(4 * (B + 1));
  L.flags = b.take(4 * B);
  L.X = b.take(2 * t_cap * d.d_model);
  L.cu = b.take(4 * (B + 1));
  L.pos = b.take(4 * t_cap);
  L.logits = b.take(sizeof(float) * static_cast<size_t>(B) * d.vocab);
  L.inner = b.off;
  const size_t a = sel_layout(d, B, nv).total, p = pack_layout(d, B, nv).total, c = pre_layout(d, B, t_cap).total;
  L.total = L.inner + std::max(a, std::max(p, c));
  return L;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

svl_status check_ws(void* ws, size_t bytes, size_t need) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255)) return SVL_ERR_WORKSPACE;
  return bytes < need ? SVL_ERR_WORKSPACE : SVL_OK;
}

GemmParams base_params(const svl_model* m) {
  GemmParams p;
  std::memset(&p, 0, sizeof(p));
  p.status = m->d_status;
  return p;
}

int gemm_grid(const svl_model* m, int64_t tiles) {
  int64_t g = std::min<int64_t>(m->num_sms, tiles);
  return static_cast<int>(std::max<int64_t>(g, 1));
}

// Counts one kernel launch and, while profiling, brackets it with a pair of
// events on its stream.
struct Launch {
  svl_model* m;
  cudaStream_t s;
  size_t first = SIZE_MAX;
  Launch(svl_model* m_, int tag, cudaStream_t s_) : m(m_), s(s_) {
    g_launches++;
    if (!m->prof || !((m->prof_mask >> tag) & 1u)) return;
    if (m->ev_used + 2 > m->ev_pool.size()) {
      for (int i = 0; i < 64; ++i) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) return;
        m->ev_pool.push_back(e);
      }
    }
    first = m->ev_used;
    m->ev_used += 2;
    m->prof_recs.emplace_back(tag, first);
    cudaEventRecord(m->ev_pool[first], s);
  }
  ~Launch() {
    if (first != SIZE_MAX) cudaEventRecord(m->ev_pool[first + 1], s);
  }
};

svl_status launch(EpiKind kind, svl_model* m, int tag, const GemmParams& p, int64_t tiles, cudaStream_t s,
                  bool e4m3 = false, bool thin = false) {
  if (tiles <= 0) return SVL_OK;
  Launch L(m, tag, s);
  return launch_gemm(kind, p, gemm_grid(m, tiles), s, e4m3, thin) == cudaSuccess ? SVL_OK : SVL_ERR_CUDA;
}

// The same for the CTA-pair kernel (QKV, gate/up): up to pair_clusters
// clusters of two, no more than the list's tiles.
svl_status launch_pair(EpiKind kind, svl_model* m, int tag, const GemmParams& p, int64_t tiles, cudaStream_t s) {
  if (tiles <= 0) return SVL_OK;
  Launch L(m, tag, s);
  const int pairs = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(m->pair_clusters, tiles)));
  return launch_gemm_pair(kind, p, pairs, s) == cudaSuccess ? SVL_OK : SVL_ERR_CUDA;
}

svl_status last_error() { return cudaGetLastError() == cudaSuccess ? SVL_OK : SVL_ERR_CUDA; }

}  // namespace

extern "C" {

const char* svl_status_string(svl_status s) {
  switch (s) {
    case SVL_OK: return "ok";
    case SVL_ERR_INVALID_ARG: return "invalid argument";
    case SVL_ERR_SHAPE: return "shape mismatch";
    case SVL_ERR_UNSUPPORTED: return "unsupported dimensions";
    case SVL_ERR_CUDA: return "CUDA error";
    case SVL_ERR_NONFINITE: return "non-finite token logit";
    case SVL_ERR_TIMEOUT: return "device wait timed out";
    case SVL_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
  }
  return "unknown status";
}

uint64_t svl_launch_count(void) { return g_launches.load(); }

int32_t svl_ksplit_plan(int32_t tiles, int32_t cap, int32_t num_sms, int32_t blocks_per_sm, int32_t units) {
  // one CTA per SM: the grid is resident at once iff an SM holds a CTA
  if (blocks_per_sm < 1) return 1;
  return ksplit_shares(tiles, cap, num_sms, units);
}

svl_status svl_model_create(const svl_model_desc* desc, const svl_weights* w, svl_model** out) {
  if (!desc || !w || !out) return SVL_ERR_INVALID_ARG;
  *out = nullptr;
  const svl_model_desc& d = *desc;
  if (d.n_layers <= 0 || d.d_model <= 0 || d.n_heads <= 0 || d.n_kv_heads <= 0 || d.d_ffn <= 0 || d.vocab <= 0 ||
      d.n_groups <= 0 || d.n_prefix < 0 || d.c_vis <= 0 || d.h_ctrl <= 0 || d.proj_hidden < 0 || d.max_seq <= 0 ||
      !(d.rms_eps > 0.f) || !(d.rope_theta > 0.f))
    return SVL_ERR_INVALID_ARG;
  if (d.d_model % d.n_heads) return SVL_ERR_UNSUPPORTED;
  const int dh = d.d_model / d.n_heads;
  const int G = d.n_groups;
  if (dh != 64 && dh != 128) return SVL_ERR_UNSUPPORTED;
  if (G > 8 || d.n_heads % G || d.n_kv_heads % G || d.n_heads % d.n_kv_heads) return SVL_ERR_UNSUPPORTED;
  if ((d.d_ffn / G) % 64 || d.d_ffn % G) return SVL_ERR_UNSUPPORTED;
  if (((d.n_heads / G) * dh) % 64) return SVL_ERR_UNSUPPORTED;
  if (d.d_model % 128 || d.c_vis % 64 || d.proj_hidden % 64) return SVL_ERR_UNSUPPORTED;
  if (d.h_ctrl % 16 || d.h_ctrl > 128) return SVL_ERR_UNSUPPORTED;
  if (d.proj_hidden == 0 && d.c_vis != d.d_model) return SVL_ERR_UNSUPPORTED;
  if (d.gemm_format != SVL_GEMM_BF16 && d.gemm_format != SVL_GEMM_E4M3) return SVL_ERR_INVALID_ARG;
  // Eq. 8 times G must stay exact in double precision at the longest sequence
  {
    const double S = d.max_seq, D = d.d_model, Dkv = static_cast<double>(d.n_kv_heads) * dh;
    const double c = G * d.n_layers * ((4 * D * D + 4 * D * Dkv + 6 * D * d.d_ffn) * S + 4 * D * S * S) +
                     G * 2.0 * D * d.vocab * S;
    if (c >= 9.0e15) return SVL_ERR_UNSUPPORTED;
  }
  if (!w->ctrl_w1 || !w->ctrl_w2 || !w->bud_w1 || !w->bud_w2 || !w->embed || !w->final_norm || !w->lm_head ||
      !w->layers)
    return SVL_ERR_INVALID_ARG;
  if (d.proj_hidden && (!w->proj_w1 || !w->proj_w2)) return SVL_ERR_INVALID_ARG;
  if (!aligned16(w->ctrl_w2) || !aligned16(w->embed)) return SVL_ERR_INVALID_ARG;  // read as 16-byte vectors
  if (!encode_fn()) return SVL_ERR_CUDA;

  svl_model* m = new svl_model();
  m->d = d;
  m->w = *w;
  m->layers.assign(w->layers, w->layers + d.n_layers);
  m->w.layers = m->layers.data();
  cudaGetDevice(&m->device);
  cudaDeviceGetAttribute(&m->num_sms, cudaDevAttrMultiProcessorCount, m->device);
  // the persistent residual GEMM runs one CTA per SM: resident at once iff
  // one CTA fits on an SM (the rule svl_ksplit_plan applies)
  m->ks_resident = gemm_resid_blocks_per_sm(d.gemm_format == SVL_GEMM_E4M3) >= 1;
  const int64_t dkv = static_cast<int64_t>(d.n_kv_heads) * dh, hq = static_cast<int64_t>(d.n_heads) * dh;
  bool ok = true;
  for (int l = 0; l < d.n_layers && ok; ++l) {
    const svl_layer_weights& lw = m->layers[l];
    ok = lw.wq && lw.wk && lw.wv && lw.wo && lw.wg && lw.wu && lw.wd && lw.attn_norm && lw.ffn_norm;
  }
  if (!ok) {
    delete m;
    return SVL_ERR_INVALID_ARG;
  }
  // RMSNorm runs fused into the GEMMs after it (x / rms(x) scales the
  // accumulator rows), so each norm gain is folded into the columns of the
  // projections it feeds: W' = W diag(gain). Layers whose gains are exactly 1
  // keep the caller's weights. e4m3 models fold nothing: their activation
  // quantiser multiplies the rows by the gain (the e4m3 definition quantises
  // RMSNorm(X) * gain and W as given), so their codes come from the caller's
  // weights.
  m->folded.assign(static_cast<size_t>(d.n_layers) * 5, nullptr);
  if (d.gemm_format != SVL_GEMM_E4M3) {
    int* flags = nullptr;
    std::vector<int> host(2 * static_cast<size_t>(d.n_layers), 1);
    ok = cudaMalloc(&flags, sizeof(int) * host.size()) == cudaSuccess &&
         cudaMemcpy(flags, host.data(), sizeof(int) * host.size(), cudaMemcpyHostToDevice) == cudaSuccess;
    for (int l = 0; l < d.n_layers && ok; ++l) {
      ok = gain_is_one(static_cast<const __nv_bfloat16*>(m->layers[l].attn_norm), d.d_model, flags + 2 * l, 0) ==
               cudaSuccess &&
           gain_is_one(static_cast<const __nv_bfloat16*>(m->layers[l].ffn_norm), d.d_model, flags + 2 * l + 1, 0) ==
               cudaSuccess;
    }
    ok = ok && cudaMemcpy(host.data(), flags, sizeof(int) * host.size(), cudaMemcpyDeviceToHost) == cudaSuccess;
    if (flags) cudaFree(flags);
    for (int l = 0; l < d.n_layers && ok; ++l) {
      svl_layer_weights& lw = m->layers[l];
      const void** src[5] = {&lw.wq, &lw.wk, &lw.wv, &lw.wg, &lw.wu};
      const int64_t rows[5] = {hq, dkv, dkv, d.d_ffn, d.d_ffn};
      for (int i = 0; i < 5 && ok; ++i) {
        const bool attn = i < 3;
        if (host[2 * l + (attn ? 0 : 1)]) continue;
        const void* gain = attn ? lw.attn_norm : lw.ffn_norm;
        void* dst = nullptr;
        ok = cudaMalloc(&dst, 2 * static_cast<size_t>(rows[i]) * d.d_model) == cudaSuccess;
        if (!ok) break;
        m->folded[static_cast<size_t>(l) * 5 + i] = dst;
        ok = fold_gain(static_cast<const __nv_bfloat16*>(*src[i]), static_cast<const __nv_bfloat16*>(gain),
                       static_cast<__nv_bfloat16*>(dst), rows[i], d.d_model, 0) == cudaSuccess;
        *src[i] = dst;
      }
    }
    if (!ok || cudaDeviceSynchronize() != cudaSuccess) {
      svl_model_destroy(m);
      return SVL_ERR_CUDA;
    }
  }
  if (d.gemm_format == SVL_GEMM_E4M3) {
    // e4m3 copies of the gated projections, one allocation per layer: codes
    // then per-row scales of q, k, v, o, g, u, d
    m->e4m3 = true;
    const int G = d.n_groups;
    m->kgo_p = round128(static_cast<int>(hq / G));
    m->kgd_p = round128(d.d_ffn / G);
    const int64_t rows[7] = {hq, dkv, dkv, d.d_model, d.d_ffn, d.d_ffn, d.d_model};
    const int groups[7] = {1, 1, 1, G, 1, 1, G};
    const int kg[7] = {d.d_model, d.d_model, d.d_model, static_cast<int>(hq / G), d.d_model, d.d_model, d.d_ffn / G};
    const int kgp[7] = {d.d_model, d.d_model, d.d_model, m->kgo_p, d.d_model, d.d_model, m->kgd_p};
    size_t code_off[7], scale_off[7], total = 0;
    for (int i = 0; i < 7; ++i) {
      code_off[i] = total;
      total = align256(total + static_cast<size_t>(rows[i]) * groups[i] * kgp[i]);
      scale_off[i] = total;
      total = align256(total + sizeof(float) * (rows[i] + 64));
    }
    m->f8_mem.assign(d.n_layers, nullptr);
    m->f8_scale.assign(static_cast<size_t>(d.n_layers) * 7, nullptr);
    m->tm8.resize(static_cast<size_t>(d.n_layers) * 7);
    for (int l = 0; l < d.n_layers && ok; ++l) {
      const svl_layer_weights& lw = m->layers[l];
      const void* src[7] = {lw.wq, lw.wk, lw.wv, lw.wo, lw.wg, lw.wu, lw.wd};
      uint8_t* base = nullptr;
      ok = cudaMalloc(&base, total) == cudaSuccess && cudaMemset(base, 0, total) == cudaSuccess;
      if (!ok) break;
      m->f8_mem[l] = base;
      for (int i = 0; i < 7 && ok; ++i) {
        QuantArgs qa;
        std::memset(&qa, 0, sizeof(qa));
        qa.src = static_cast<const __nv_bfloat16*>(src[i]);
        qa.ld_src = static_cast<int64_t>(groups[i]) * kg[i];
        qa.rows = rows[i];
        qa.G = groups[i];
        qa.kg = kg[i];
        qa.kgp = kgp[i];
        qa.dst = base + code_off[i];
        qa.ld_dst = static_cast<int64_t>(groups[i]) * kgp[i];
        qa.scale = reinterpret_cast<float*>(base + scale_off[i]);
        m->f8_scale[static_cast<size_t>(l) * 7 + i] = qa.scale;
        ok = launch_quant_rows(qa, 0) == cudaSuccess &&
             make_map8(&m->tm8[static_cast<size_t>(l) * 7 + i], qa.dst, rows[i], qa.ld_dst);
        g_launches++;
      }
    }
    if (!ok || cudaDeviceSynchronize() != cudaSuccess) {
      svl_model_destroy(m);
      return SVL_ERR_CUDA;
    }
  }
  m->tm_layer.resize(static_cast<size_t>(d.n_layers) * 7);
  for (int l = 0; l < d.n_layers && ok; ++l) {
    const svl_layer_weights& lw = m->layers[l];
    CUtensorMap* t = &m->tm_layer[static_cast<size_t>(l) * 7];
    ok = make_map(t + 0, lw.wq, hq, d.d_model) && make_map(t + 1, lw.wk, dkv, d.d_model) &&
         make_map(t + 2, lw.wv, dkv, d.d_model) && make_map(t + 3, lw.wo, d.d_model, hq) &&
         make_map(t + 4, lw.wg, d.d_ffn, d.d_model) && make_map(t + 5, lw.wu, d.d_ffn, d.d_model) &&
         make_map(t + 6, lw.wd, d.d_model, d.d_ffn);
  }
  ok = ok && make_map(&m->tm_ctrl_w1, w->ctrl_w1, d.h_ctrl, d.c_vis, static_cast<uint32_t>(d.h_ctrl)) &&
       make_map(&m->tm_lm_head, w->lm_head, d.vocab, d.d_model);
  if (ok && d.proj_hidden)
    ok = make_map(&m->tm_proj_w1, w->proj_w1, d.proj_hidden, d.c_vis) &&
         make_map(&m->tm_proj_w2, w->proj_w2, d.d_model, d.proj_hidden);
  if (!ok) {
    svl_model_destroy(m);
    return SVL_ERR_INVALID_ARG;
  }
  // CTA-pair QKV and gate/up GEMMs for bf16 models, chosen with
  // SVL_PAIR_GEMM=1 in the environment at model creation. They move a third
  // less data through shared memory and L2 per FLOP but run at the same speed
  // as the single-CTA kernel on GB300, whose GEMMs are held by the power cap,
  // so the single-CTA kernel stays the default.
  if (ok && !m->e4m3) {
    const char* env = std::getenv("SVL_PAIR_GEMM");
    if (env && env[0] == '1') {
      const int c = std::min(gemm_pair_max_clusters(EPI_QKV_ROPE), gemm_pair_max_clusters(EPI_SWIGLU));
      m->pair_clusters = std::min(c, m->num_sms / 2);
    }
    cudaGetLastError();  // a failed occupancy query only disables the pair kernel
    if (m->pair_clusters > 0) {
      m->tm_pair.resize(static_cast<size_t>(d.n_layers) * 5);
      for (int l = 0; l < d.n_layers && ok; ++l) {
        const svl_layer_weights& lw = m->layers[l];
        CUtensorMap* t = &m->tm_pair[static_cast<size_t>(l) * 5];
        ok = make_map(t + 0, lw.wq, hq, d.d_model, 64) && make_map(t + 1, lw.wk, dkv, d.d_model, 64) &&
             make_map(t + 2, lw.wv, dkv, d.d_model, 64) && make_map(t + 3, lw.wg, d.d_ffn, d.d_model, 64) &&
             make_map(t + 4, lw.wu, d.d_ffn, d.d_model, 64);
      }
      if (!ok) {
        svl_model_destroy(m);
        return SVL_ERR_INVALID_ARG;
      }
    }
  }
  if (cudaMalloc(&m->d_status, sizeof(uint32_t)) != cudaSuccess ||
      cudaMalloc(&m->rope_cs, sizeof(float2) * static_cast<size_t>(d.max_seq) * (dh / 2)) != cudaSuccess) {
    svl_model_destroy(m);
    return SVL_ERR_CUDA;
  }
  cudaMemset(m->d_status, 0, sizeof(uint32_t));
  launch_rope_table(m->rope_cs, d.max_seq, dh, static_cast<double>(d.rope_theta), 0);
  g_launches++;
  if (cudaDeviceSynchronize() != cudaSuccess) {
    svl_model_destroy(m);
    return SVL_ERR_CUDA;
  }
  *out = m;
  return SVL_OK;
}

void svl_model_destroy(svl_model* m) {
  if (!m) return;
  for (cudaEvent_t e : m->ev_pool) cudaEventDestroy(e);
  if (m->d_status) cudaFree(m->d_status);
  if (m->rope_cs) cudaFree(m->rope_cs);
  for (void* f : m->folded)
    if (f) cudaFree(f);
  for (void* f : m->f8_mem)
    if (f) cudaFree(f);
  delete m;
}

size_t svl_workspace_size_for(const svl_model* m, uint32_t stages, int32_t max_batch, int64_t max_vis_total,
                              int64_t max_text_total) {
  if (!m || max_batch <= 0 || max_vis_total < 0 || max_text_total < 0) return 0;
  size_t need = 0;
  if (stages & SVL_STAGE_SELECT) need = std::max(need, sel_layout(m->d, max_batch, max_vis_total).total);
  if (stages & SVL_STAGE_PACK) need = std::max(need, pack_layout(m->d, max_batch, max_vis_total).total);
  if (stages & SVL_STAGE_PREFILL)
    need = std::max(need, pre_layout(m->d, max_batch, max_vis_total + max_text_total + max_batch).total);
  return need;
}

size_t svl_workspace_size(const svl_model* m, int32_t max_batch, int64_t max_vis_total, int64_t max_text_total) {
  return svl_workspace_size_for(m, SVL_STAGE_SELECT | SVL_STAGE_PACK | SVL_STAGE_PREFILL, max_batch, max_vis_total,
                                max_text_total);
}

namespace {
// Token controller: scores, k and the kept lists. Gates are given
// (layer_gate, group_gate) or, under the paper's rule, derived from the
// compute controller's logits and projected (gate_logits, *_out).
svl_status score_select_impl(svl_model* m, int32_t B, int32_t n_vis_total, const void* vis_feats,
                             const int32_t* vis_off, const int32_t* text_len, const float* budget,
                             const int32_t* keep_count, const uint8_t* layer_gate, const uint8_t* group_gate,
                             int rule, const float* gate_logits, uint8_t* layer_gate_out, uint8_t* group_gate_out,
                             float* kappa_out, float* scores, int32_t* k, int32_t* kept_idx, int32_t* kept_off,
                             uint32_t* sample_flags, void* ws, size_t ws_bytes, void* stream) {
  // rule 0: budget count for given gates; 1: paper rule with gate logits;
  // 2: paper rule, gates decided later (threshold only)
  if (!m || B <= 0 || n_vis_total < 0 || !vis_off || !text_len || !budget || !scores || !k || !kept_idx || !kept_off)
    return SVL_ERR_INVALID_ARG;
  if (rule == 0 && (!layer_gate || !group_gate)) return SVL_ERR_INVALID_ARG;
  if (rule == 1 && (!gate_logits || !layer_gate_out || !group_gate_out)) return SVL_ERR_INVALID_ARG;
  if (n_vis_total > 0 && (!vis_feats || !aligned16(vis_feats))) return SVL_ERR_INVALID_ARG;
  const SelLayout L = sel_layout(m->d, B, n_vis_total);
  svl_status st = check_ws(ws, ws_bytes, L.total);
  if (st != SVL_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const svl_model_desc& d = m->d;
  float* e_b = at<float>(ws, L.e_b);

  {
    Launch L(m, SVL_TAG_BUDGET_EMBED, s);
    launch_budget_embed(budget, static_cast<const __nv_bfloat16*>(m->w.bud_w1),
                        static_cast<const __nv_bfloat16*>(m->w.bud_w2), d.h_ctrl, B, e_b, s);
  }

  if (n_vis_total > 0) {
    GemmParams p = base_params(m);
    if (!make_map(&p.mapA, vis_feats, n_vis_total, d.c_vis)) return SVL_ERR_INVALID_ARG;
    p.mapB[0] = m->tm_ctrl_w1;
    p.grid_m = (n_vis_total + kBM - 1) / kBM;
    p.grid_n = 1;
    p.bn = d.h_ctrl;
    p.m_limit = n_vis_total;
    p.n_limit = d.h_ctrl;
    p.K = d.c_vis;
    p.kgroup = d.c_vis;
    p.out[0] = scores;
    p.e_b = e_b;
    p.seg_off = vis_off;
    p.n_seg = B;
    p.w2 = static_cast<const __nv_bfloat16*>(m->w.ctrl_w2);
    p.c2 = m->w.ctrl_c2;
    p.b_box_rows = d.h_ctrl;
    st = launch(d.h_ctrl <= 64 ? EPI_SCORE : EPI_SCORE_WIDE, m, SVL_TAG_SCORE, p, p.grid_m, s);
    if (st != SVL_OK) return st;
  }

  SelectArgs a;
  std::memset(&a, 0, sizeof(a));
  a.scores = scores;
  a.vis_off = vis_off;
  a.text_len = text_len;
  a.budget = budget;
  a.keep_count = keep_count;
  a.layer_gate = layer_gate;
  a.group_gate = group_gate;
  a.L = d.n_layers;
  a.G = d.n_groups;
  a.P = d.n_prefix;
  a.D = d.d_model;
  a.Dkv = static_cast<long long>(d.n_kv_heads) * (d.d_model / d.n_heads);
  a.Di = d.d_ffn;
  a.V = d.vocab;
  a.k_out = k;
  a.flags = sample_flags;
  a.kept_local = at<int>(ws, L.kept_local);
  a.gate_logits = rule == 1 ? gate_logits : nullptr;
  a.layer_gate_out = layer_gate_out;
  a.group_gate_out = group_gate_out;
  a.threshold_only = rule == 2 ? 1 : 0;
  a.kappa = kappa_out;
  {
    Launch L1(m, SVL_TAG_SELECT, s);
    launch_select(a, B, s);
  }
  {
    Launch L2(m, SVL_TAG_SELECT, s);
    launch_compact(B, vis_off, k, a.kept_local, kept_idx, kept_off, at<int>(ws, L.scalars), s);
  }
  return last_error();
}
}  // namespace

svl_status svl_score_select(svl_model* m, int32_t B, int32_t n_vis_total, const void* vis_feats,
                            const int32_t* vis_off, const int32_t* text_len, const float* budget,
                            const int32_t* keep_count, const uint8_t* layer_gate, const uint8_t* group_gate,
                            float* scores, int32_t* k, int32_t* kept_idx, int32_t* kept_off, uint32_t* sample_flags,
                            void* ws, size_t ws_bytes, void* stream) {
  return score_select_impl(m, B, n_vis_total, vis_feats, vis_off, text_len, budget, keep_count, layer_gate,
                           group_gate, 0, nullptr, nullptr, nullptr, nullptr, scores, k, kept_idx, kept_off,
                           sample_flags, ws, ws_bytes, stream);
}

svl_status svl_score_select_paper(svl_model* m, int32_t B, int32_t n_vis_total, const void* vis_feats,
                                  const int32_t* vis_off, const int32_t* text_len, const float* budget,
                                  const int32_t* keep_count, const float* gate_logits, float* scores, int32_t* k,
                                  int32_t* kept_idx, int32_t* kept_off, uint32_t* sample_flags,
                                  uint8_t* layer_gate_out, uint8_t* group_gate_out, float* kappa_out, void* ws,
                                  size_t ws_bytes, void* stream) {
  return score_select_impl(m, B, n_vis_total, vis_feats, vis_off, text_len, budget, keep_count, nullptr, nullptr,
                           gate_logits ? 1 : 2, gate_logits, layer_gate_out, group_gate_out, kappa_out, scores, k,
                           kept_idx, kept_off, sample_flags, ws, ws_bytes, stream);
}

namespace {
// Packs kept visual rows and text rows; with `budget` (compute controller,
// Sec. 3.2) each sample also gets its budget token as its last row.
svl_status pack_impl(svl_model* m, int32_t B, int32_t n_vis_total, int32_t n_text_total, const void* vis_feats,
                     const int32_t* vis_off, const int32_t* kept_idx, const int32_t* kept_off,
                     const int32_t* text_ids, const int32_t* text_off, const float* budget, void* X,
                     int32_t* cu_seqlens, int32_t* pos, void* ws, size_t ws_bytes, void* stream) {
  if (!m || B <= 0 || n_vis_total < 0 || n_text_total < 0 || !vis_off || !kept_idx || !kept_off || !text_off ||
      !X || !cu_seqlens || !pos)
    return SVL_ERR_INVALID_ARG;
  if ((n_text_total > 0 && !text_ids) || (n_vis_total > 0 && !vis_feats)) return SVL_ERR_INVALID_ARG;
  if (!aligned16(X) || (vis_feats && !aligned16(vis_feats))) return SVL_ERR_INVALID_ARG;
  const PackLayout L = pack_layout(m->d, B, n_vis_total);
  svl_status st = check_ws(ws, ws_bytes, L.total);
  if (st != SVL_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const svl_model_desc& d = m->d;
  const int64_t t_cap = static_cast<int64_t>(n_vis_total) + n_text_total + (budget ? B : 0);
  if (t_cap > INT32_MAX / 2) return SVL_ERR_SHAPE;

  PackArgs a;
  std::memset(&a, 0, sizeof(a));
  if (budget) {
    __nv_bfloat16* tok = at<__nv_bfloat16>(ws, L.tok);
    a.tok_rows = tok;
    Launch L0(m, SVL_TAG_PACK, s);
    launch_llm_budget_embed(budget, static_cast<const __nv_bfloat16*>(m->w.llm_bud_w1),
                            static_cast<const __nv_bfloat16*>(m->w.llm_bud_w2), d.h_ctrl, d.d_model, B, tok, s);
  }
  a.B = B;
  a.D = d.d_model;
  a.c_vis = d.c_vis;
  a.V = d.vocab;
  a.t_cap = static_cast<int>(t_cap);
  a.vis = static_cast<const __nv_bfloat16*>(vis_feats);
  a.vis_off = vis_off;
  a.kept_idx = kept_idx;
  a.kept_off = kept_off;
  a.text_ids = text_ids;
  a.text_off = text_off;
  a.embed = static_cast<const __nv_bfloat16*>(m->w.embed);
  a.X = static_cast<__nv_bfloat16*>(X);
  a.cu_seqlens = cu_seqlens;
  a.pos = pos;
  a.t_total = at<int>(ws, L.scalars) + 1;
  a.use_projector = d.proj_hidden ? 1 : 0;
  a.stage = d.proj_hidden ? at<__nv_bfloat16>(ws, L.stage) : nullptr;
  a.row_map = d.proj_hidden ? at<int>(ws, L.row_map) : nullptr;
  a.status = m->d_status;
  {
    Launch L1(m, SVL_TAG_PACK, s);
    launch_pack_offsets(a, s);
  }
  {
    Launch L2(m, SVL_TAG_PACK, s);
    launch_pack_gather(a, s);
  }

  if (d.proj_hidden && n_vis_total > 0) {
    GemmParams p = base_params(m);
    if (!make_map(&p.mapA, a.stage, n_vis_total, d.c_vis)) return SVL_ERR_CUDA;
    p.mapB[0] = m->tm_proj_w1;
    p.grid_m = (n_vis_total + kBM - 1) / kBM;
    p.grid_n = (d.proj_hidden + 255) / 256;
    p.bn = 256;
    p.m_limit_dev = kept_off + B;
    p.m_limit = n_vis_total;
    p.n_limit = d.proj_hidden;
    p.K = d.c_vis;
    p.kgroup = d.c_vis;
    p.out[0] = at<__nv_bfloat16>(ws, L.hp);
    p.ld[0] = d.proj_hidden;
    st = launch(EPI_GELU, m, SVL_TAG_PROJECTOR, p, static_cast<int64_t>(p.grid_m) * p.grid_n, s);
    if (st != SVL_OK) return st;

    GemmParams q = base_params(m);
    if (!make_map(&q.mapA, at<__nv_bfloat16>(ws, L.hp), n_vis_total, d.proj_hidden)) return SVL_ERR_CUDA;
    q.mapB[0] = m->tm_proj_w2;
    q.grid_m = p.grid_m;
    q.grid_n = (d.d_model + 255) / 256;
    q.bn = 256;
    q.m_limit_dev = kept_off + B;
    q.m_limit = n_vis_total;
    q.n_limit = d.d_model;
    q.K = d.proj_hidden;
    q.kgroup = d.proj_hidden;
    q.out[0] = X;
    q.ld[0] = d.d_model;
    q.row_map = a.row_map;
    st = launch(EPI_ROWMAP, m, SVL_TAG_PROJECTOR, q, static_cast<int64_t>(q.grid_m) * q.grid_n, s);
    if (st != SVL_OK) return st;
  }
  return last_error();
}
}  // namespace

svl_status svl_pack(svl_model* m, int32_t B, int32_t n_vis_total, int32_t n_text_total, const void* vis_feats,
                    const int32_t* vis_off, const int32_t* kept_idx, const int32_t* kept_off,
                    const int32_t* text_ids, const int32_t* text_off, void* X, int32_t* cu_seqlens, int32_t* pos,
                    void* ws, size_t ws_bytes, void* stream) {
  return pack_impl(m, B, n_vis_total, n_text_total, vis_feats, vis_off, kept_idx, kept_off, text_ids, text_off,
                   nullptr, X, cu_seqlens, pos, ws, ws_bytes, stream);
}

svl_status svl_pack_controlled(svl_model* m, int32_t B, int32_t n_vis_total, int32_t n_text_total,
                               const void* vis_feats, const int32_t* vis_off, const int32_t* kept_idx,
                               const int32_t* kept_off, const int32_t* text_ids, const int32_t* text_off,
                               const float* budget, void* X, int32_t* cu_seqlens, int32_t* pos, void* ws,
                               size_t ws_bytes, void* stream) {
  if (!m || !budget) return SVL_ERR_INVALID_ARG;
  if (!m->w.llm_bud_w1 || !m->w.llm_bud_w2) return SVL_ERR_UNSUPPORTED;
  return pack_impl(m, B, n_vis_total, n_text_total, vis_feats, vis_off, kept_idx, kept_off, text_ids, text_off,
                   budget, X, cu_seqlens, pos, ws, ws_bytes, stream);
}

namespace {
// One stage of one layer on caller buffers (svl_layer_stage): the stage's
// inputs and outputs replace the workspace copies of Q, K, V^T, the
// attention output and the SwiGLU output.
struct StageSel {
  int stage, layer;
  __nv_bfloat16 *q, *k, *vt, *ao, *h;
};

// KV cache of a prefill (store each layer's K, V) or a decode step (one new
// row per sample: embedding of the fed token, attention against the cache,
// greedy next token).
struct StepCtx {
  __nv_bfloat16* kv;  // [2][L][B][max_len][dkv]
  int max_len;
  int decode;
  int* cache_len;        // [B] decode: positions so far (advanced by one)
  const int* tokens;     // [B] decode: fed token ids
  int* next_token;       // [B] decode: greedy next token, or nullptr
};

// The gated decoder forward. With `ctl` (compute controller, Sec. 3.2) the
// gate arrays are outputs: they start all on, the controller kernel writes
// them after the prefix layers, and the device schedule is built again.
// With `kvx` the keys and values go to the cache (prefill) or the step is a
// decode step over one row per sample.
svl_status prefill_impl(svl_model* m, int32_t B, int32_t t_cap, void* X, const int32_t* cu_seqlens,
                        const int32_t* pos, const uint8_t* layer_gate, const uint8_t* group_gate,
                        int32_t logits_mode, float* logits, void* ws, size_t ws_bytes, void* stream,
                        const CtlArgs* ctl, const StepCtx* kvx = nullptr, const StageSel* only = nullptr) {
  if (!m || B <= 0 || t_cap <= 0 || !X || !cu_seqlens || !pos || !layer_gate || !group_gate || (!logits && !only))
    return SVL_ERR_INVALID_ARG;
  if (logits_mode != SVL_LOGITS_LAST && logits_mode != SVL_LOGITS_ALL) return SVL_ERR_INVALID_ARG;
  if (!aligned16(X)) return SVL_ERR_INVALID_ARG;
  if (B > kMaxPrefillBatch) return SVL_ERR_UNSUPPORTED;  // the schedule stages per-sample data in shared memory
  const PreLayout L = pre_layout(m->d, B, t_cap);
  svl_status st = check_ws(ws, ws_bytes, L.total);
  if (st != SVL_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const svl_model_desc& d = m->d;
  const int dh = d.d_model / d.n_heads;
  const int hq = d.n_heads * dh, dkv = d.n_kv_heads * dh;
  const int nl = d.n_layers;
  int* counts = at<int>(ws, L.counts);
  if (kvx && kvx->decode) {
    // the step's rows: embeddings of the fed tokens at their cache positions
    Launch L0(m, SVL_TAG_PACK, s);
    launch_decode_prep(B, d.d_model, d.vocab, kvx->tokens, kvx->cache_len, kvx->max_len,
                       static_cast<const __nv_bfloat16*>(m->w.embed), static_cast<__nv_bfloat16*>(X),
                       const_cast<int32_t*>(cu_seqlens), const_cast<int32_t*>(pos), m->d_status, s);
  }

  ScheduleArgs sa;
  sa.B = B;
  sa.L = nl;
  sa.G = d.n_groups;
  sa.P = d.n_prefix;
  sa.num_sms = m->num_sms;
  const bool thin_launch = t_cap <= kThinRows;
  const bool pair = m->pair_clusters > 0 && !m->e4m3 && !thin_launch;
  sa.nsparse_rows = pair ? 2 * kBM : kBM;
  sa.nsparse_wave = pair ? m->pair_clusters : m->num_sms;
  sa.A = d.n_heads;
  sa.Akv = d.n_kv_heads;
  sa.dh = dh;
  sa.D = d.d_model;
  sa.Di = d.d_ffn;
  {
    const long long row_bytes = static_cast<long long>(sa.nsparse_rows) * d.d_model * (m->e4m3 ? 1 : 2);
    sa.mband = static_cast<int>(std::max<long long>(1, kMBandBytes / row_bytes));
  }
  sa.cu_seqlens = cu_seqlens;
  sa.layer_gate = layer_gate;
  sa.group_gate = group_gate;
  sa.act = at<uint8_t>(ws, L.act);
  sa.seg = at<int4>(ws, L.seg);
  sa.qkv_tiles = at<int4>(ws, L.qkv);
  sa.qkv_cap = L.qkv_cap;
  sa.qkv_count = counts;
  sa.o_tiles = at<int4>(ws, L.o);
  sa.o_cap = L.o_cap;
  sa.o_count = counts + nl;
  sa.gu_tiles = at<int4>(ws, L.gu);
  sa.gu_cap = L.gu_cap;
  sa.gu_count = counts + 2 * nl;
  sa.dn_tiles = at<int4>(ws, L.dn);
  sa.dn_cap = L.dn_cap;
  sa.dn_count = counts + 3 * nl;
  sa.attn_items = at<int4>(ws, L.attn);
  sa.attn_cap = L.attn_cap;
  sa.attn_count = counts + 4 * nl;
  sa.attn_next = counts + 5 * nl;
  sa.ks_info = at<int>(ws, L.ks_info);
  sa.ks_units = m->ks_resident ? L.ks_units : 0;
  sa.status = m->d_status;
  if (ctl) {
    // controller path: every group on until the controller has decided
    if (cudaMemsetAsync(const_cast<uint8_t*>(layer_gate), 1, static_cast<size_t>(B) * nl, s) != cudaSuccess ||
        cudaMemsetAsync(const_cast<uint8_t*>(group_gate), 1, static_cast<size_t>(B) * nl * d.n_groups, s) !=
            cudaSuccess)
      return SVL_ERR_CUDA;
  }
  int* ks_ticket = at<int>(ws, L.ks_ticket);
  if (cudaMemsetAsync(ks_ticket, 0, sizeof(int) * L.ks_units * 2 * nl, s) != cudaSuccess) return SVL_ERR_CUDA;
  {
    Launch L1(m, SVL_TAG_SCHEDULE, s);
    launch_schedule(sa, s);
  }

  __nv_bfloat16* xn = at<__nv_bfloat16>(ws, L.xn);
  __nv_bfloat16* qb = only ? only->q : at<__nv_bfloat16>(ws, L.q);
  __nv_bfloat16* kb = only ? only->k : at<__nv_bfloat16>(ws, L.k);
  __nv_bfloat16* vb = only ? only->vt : at<__nv_bfloat16>(ws, L.v);
  __nv_bfloat16* ao = only ? only->ao : at<__nv_bfloat16>(ws, L.ao);
  __nv_bfloat16* hm = only ? only->h : at<__nv_bfloat16>(ws, L.hmid);
  // decode-sized batches (one row per sample) stream the weights through the
  // gated GEMMs with A boxes of kThinRows rows and deeper stages
  const bool thin = t_cap <= kThinRows;
  const uint32_t a_rows = thin ? kThinRows : 128;
  CUtensorMap map_x, map_xn, map_ao, map_hm, map_xr, map_hmo;
  if (!make_map(&map_x, X, t_cap, d.d_model, a_rows) || !make_map(&map_xn, xn, t_cap, d.d_model) ||
      !make_map(&map_ao, ao, t_cap, hq, a_rows) || !make_map(&map_hm, hm, t_cap, d.d_ffn, a_rows) ||
      !make_map(&map_xr, X, t_cap, d.d_model, 32) ||  // residual stream, 32-row boxes (residual epilogues)
      !make_map(&map_hmo, hm, t_cap, d.d_ffn, 32))    // SwiGLU outputs, 32-row boxes (gate/up epilogue)
    return SVL_ERR_CUDA;
  CUtensorMap map_q32, map_k32;  // Q and K, 32-row boxes (QKV epilogue)
  if (!make_map(&map_q32, qb, t_cap, hq, 32) || !make_map(&map_k32, kb, t_cap, dkv, 32)) return SVL_ERR_CUDA;
  // e4m3: every gated GEMM reads the quantised rows of its input (aq, with
  // per-row scales as) -- X for QKV and gate/up, the attention output for
  // O, the SwiGLU output for down (both group-padded to whole K blocks)
  const bool f8 = m->e4m3;
  const int G = d.n_groups;
  uint8_t* aq = f8 ? at<uint8_t>(ws, L.aq) : nullptr;
  float* as = f8 ? at<float>(ws, L.as) : nullptr;
  CUtensorMap map_aq_x, map_aq_o, map_aq_h;
  if (f8 && (!make_map8(&map_aq_x, aq, t_cap, d.d_model, a_rows) ||
             !make_map8(&map_aq_o, aq, t_cap, static_cast<uint64_t>(G) * m->kgo_p, a_rows) ||
             !make_map8(&map_aq_h, aq, t_cap, static_cast<uint64_t>(G) * m->kgd_p, a_rows)))
    return SVL_ERR_CUDA;
  auto quant = [&](const __nv_bfloat16* src, const void* gain, int64_t ld_src, int groups, int kg, int kgp,
                   int layer) {
    QuantArgs qa;
    std::memset(&qa, 0, sizeof(qa));
    qa.src = src;
    qa.gain = static_cast<const __nv_bfloat16*>(gain);
    qa.ld_src = ld_src;
    qa.rows = t_cap;
    qa.G = groups;
    qa.kg = kg;
    qa.kgp = kgp;
    qa.dst = aq;
    qa.ld_dst = static_cast<int64_t>(groups) * kgp;
    qa.scale = as;
    qa.cu_seqlens = cu_seqlens;
    qa.B = B;
    if (layer >= 0) {
      qa.layer_gate = layer_gate;
      qa.group_gate = group_gate;
      qa.L = nl;
      qa.l = layer;
      qa.P = d.n_prefix;
    }
    Launch L1(m, SVL_TAG_QUANT, s);
    return launch_quant_rows(qa, s) == cudaSuccess ? SVL_OK : SVL_ERR_CUDA;
  };
  auto set_f8 = [&](GemmParams& p, const CUtensorMap& mapA, const CUtensorMap* tm8, const float* const* sc,
                    std::initializer_list<int> mats) {
    p.mapA = mapA;
    int i = 0;
    for (int mat : mats) {
      p.mapB[i] = tm8[mat];
      p.b_scale[i] = sc[mat];
      ++i;
    }
    p.a_scale = as;
  };

  // fused RMSNorm: per-row partial sums of squares of X (see GemmParams)
  float* ss_a = at<float>(ws, L.ss_a);
  float* ss_b = at<float>(ws, L.ss_b);
  const int ss_ld = static_cast<int>(L.t_pad);
  auto set_norm = [&](GemmParams& p, const float* in, float* out) {
    p.ss_in = in;
    p.ss_out = out;
    p.ss_ld = ss_ld;
    p.ss_slots = L.ss_slots;
    p.ss_inv_d = 1.f / static_cast<float>(d.d_model);
    p.ss_eps = d.rms_eps;
  };

  NormArgs na;
  na.t_cap = t_cap;
  na.D = d.d_model;
  na.B = B;
  na.eps = d.rms_eps;
  na.X = static_cast<const __nv_bfloat16*>(X);
  na.Y = xn;
  na.cu_seqlens = cu_seqlens;

  // V^T is read in 128-key tiles that may run past the rows written in this
  // call; zero it once so those (masked) keys hold finite values (a single
  // stage reads or writes the caller's V^T as it is)
  if (!only && cudaMemsetAsync(vb, 0, sizeof(__nv_bfloat16) * static_cast<size_t>(L.t_pad) * dkv, s) != cudaSuccess)
    return SVL_ERR_CUDA;
  AttnTcArgs aa;
  std::memset(&aa, 0, sizeof(aa));
  if (!make_map(&aa.mapQ, qb, t_cap, hq) || !make_map(&aa.mapVt, vb, dkv, L.t_pad, static_cast<uint32_t>(dh)) ||
      !make_map(&aa.mapK64, kb, t_cap, dkv, 64) || !make_map(&aa.mapO, ao, t_cap, hq, 32))
    return SVL_ERR_CUDA;
  aa.cap = L.attn_cap;
  aa.A = d.n_heads;
  aa.Akv = d.n_kv_heads;
  aa.dh = dh;
  aa.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(dh)));
  aa.O = ao;
  aa.ldo = hq;
  aa.status = m->d_status;

  {
    // sums of squares of the input rows: for the first layer's attention
    // norm, or for the MLP norm when a single gate/up stage runs
    Launch L1(m, SVL_TAG_RMSNORM, s);
    launch_norm_init(static_cast<const __nv_bfloat16*>(X), cu_seqlens, B, static_cast<int>(t_cap), d.d_model,
                     only && only->stage == SVL_LAYER_GATEUP ? ss_b : ss_a, ss_ld, L.ss_slots, s);
  }
  // a stage of the layer runs unless a single other stage was asked for
  auto want = [&](int l, int stage) { return !only || (only->layer == l && only->stage == stage); };

  for (int l = 0; l < nl; ++l) {
    if (only && l != only->layer) continue;
    const CUtensorMap* tm = &m->tm_layer[static_cast<size_t>(l) * 7];
    if (ctl && l == std::min(d.n_prefix, nl)) {
      // the budget token's state after the prefix layers decides the gates
      // of the remaining layers; their tile lists are rebuilt on the device
      CtlArgs c = *ctl;
      c.X = static_cast<const __nv_bfloat16*>(X);
      c.cu_seqlens = cu_seqlens;
      c.layer_gate = const_cast<uint8_t*>(layer_gate);
      c.group_gate = const_cast<uint8_t*>(group_gate);
      {
        Launch L1(m, SVL_TAG_SCHEDULE, s);
        launch_controller(c, s);
      }
      {
        Launch L1(m, SVL_TAG_SCHEDULE, s);
        launch_schedule(sa, s);
      }
    }

    const CUtensorMap* tm8 = f8 ? &m->tm8[static_cast<size_t>(l) * 7] : nullptr;
    const float* const* sc8 = f8 ? &m->f8_scale[static_cast<size_t>(l) * 7] : nullptr;
    GemmParams p;
    if (want(l, SVL_LAYER_QKV)) {
    // attention input norm fused into the QKV GEMM (bf16: gain folded into
    // W_qkv; e4m3: the quantiser multiplies the rows by the gain)
    if (f8 && (st = quant(static_cast<const __nv_bfloat16*>(X), m->layers[l].attn_norm, d.d_model, 1, d.d_model,
                          d.d_model, -1)) != SVL_OK)
      return st;
    p = base_params(m);
    set_norm(p, ss_a, nullptr);
    p.mapA = map_x;
    p.mapB[0] = tm[0];
    p.mapB[1] = tm[1];
    p.mapB[2] = tm[2];
    if (f8) set_f8(p, map_aq_x, tm8, sc8, {0, 1, 2});
    if (pair) {
      const CUtensorMap* tp = &m->tm_pair[static_cast<size_t>(l) * 5];
      p.mapB[0] = tp[0];
      p.mapB[1] = tp[1];
      p.mapB[2] = tp[2];
    }
    p.tiles = sa.qkv_tiles + static_cast<size_t>(l) * L.qkv_cap;
    p.tile_count = counts + l;
    p.max_tiles = L.qkv_cap;
    p.K = d.d_model;
    p.kgroup = d.d_model;
    p.out[0] = qb;
    p.out[1] = kb;
    p.out[2] = vb;
    p.ld[0] = hq;
    p.ld[1] = dkv;
    p.ld[2] = static_cast<int>(L.t_pad);
    p.pos = pos;
    p.rope_cs = m->rope_cs;
    p.rope_rows = d.max_seq;
    p.d_head = dh;
    p.mapR = map_q32;
    p.mapR2 = map_k32;
    p.stage_tma = 1;
    if ((st = pair ? launch_pair(EPI_QKV_ROPE, m, SVL_TAG_QKV, p, L.qkv_cap, s)
                   : launch(EPI_QKV_ROPE, m, SVL_TAG_QKV, p, L.qkv_cap, s, f8, thin)) != SVL_OK)
      return st;
    }

    if (want(l, SVL_LAYER_ATTN)) {
    const size_t layer_kv = static_cast<size_t>(B) * (kvx ? kvx->max_len : 0) * dkv;
    if (kvx && kvx->decode) {
      DecAttnArgs da;
      std::memset(&da, 0, sizeof(da));
      da.B = B;
      da.A = d.n_heads;
      da.Akv = d.n_kv_heads;
      da.dh = dh;
      da.dkv = dkv;
      da.G = d.n_groups;
      da.L = nl;
      da.P = d.n_prefix;
      da.l = l;
      da.max_len = kvx->max_len;
      da.t_pad = static_cast<int>(L.t_pad);
      da.ldq = hq;
      da.ldo = hq;
      da.scale = static_cast<float>(1.0 / std::sqrt(static_cast<double>(dh)));
      da.cache_len = kvx->cache_len;
      da.layer_gate = layer_gate;
      da.group_gate = group_gate;
      da.q = qb;
      da.k = kb;
      da.vt = vb;
      da.k_cache = kvx->kv + static_cast<size_t>(l) * layer_kv;
      da.v_cache = kvx->kv + static_cast<size_t>(nl + l) * layer_kv;
      da.out = ao;
      Launch L1(m, SVL_TAG_ATTENTION, s);
      launch_decode_attn(da, s);
    } else {
      if (kvx) {
        KvArgs ka;
        ka.B = B;
        ka.dkv = dkv;
        ka.max_len = kvx->max_len;
        ka.t_pad = static_cast<int>(L.t_pad);
        ka.cu_seqlens = cu_seqlens;
        ka.pos = pos;
        ka.k = kb;
        ka.vt = vb;
        ka.k_cache = kvx->kv + static_cast<size_t>(l) * layer_kv;
        ka.v_cache = kvx->kv + static_cast<size_t>(nl + l) * layer_kv;
        Launch L1(m, SVL_TAG_COPY, s);
        launch_kv_store(ka, t_cap, s);
      }
      aa.items = sa.attn_items + static_cast<size_t>(l) * L.attn_cap;
      aa.count = counts + 4 * nl + l;
      aa.next_unit = counts + 5 * nl + l;
      Launch L1(m, SVL_TAG_ATTENTION, s);
      if (launch_attention_tc(aa, gemm_grid(m, L.attn_cap), s) != cudaSuccess) return SVL_ERR_CUDA;
    }
    }

    if (want(l, SVL_LAYER_OPROJ)) {
    if (f8 && (st = quant(ao, nullptr, hq, G, hq / G, m->kgo_p, l)) != SVL_OK) return st;
    p = base_params(m);
    p.mapA = map_ao;
    p.mapB[0] = tm[3];
    p.tiles = sa.o_tiles + static_cast<size_t>(l) * L.o_cap;
    p.tile_count = counts + nl + l;
    p.max_tiles = L.o_cap;
    p.K = hq;
    p.kgroup = hq / d.n_groups;
    if (f8) {
      set_f8(p, map_aq_o, tm8, sc8, {3});
      p.K = G * m->kgo_p;
      p.kgroup = m->kgo_p;
    }
    p.out[0] = X;
    p.ld[0] = d.d_model;
    p.mapR = map_xr;
    p.stage_tma = 1;
    p.a_evict_first = 1;  // n-band list: the weights stay in L2, the input rows stream
    p.ks_info = sa.ks_info + static_cast<size_t>(l) * 8;
    p.ks_part = at<float>(ws, L.ks_part);
    p.ks_ticket = ks_ticket + static_cast<size_t>(2 * l) * L.ks_units;
    set_norm(p, nullptr, ss_b);  // sums of squares of the updated rows for the MLP norm
    if ((st = launch(EPI_RESID, m, SVL_TAG_OPROJ, p, L.o_cap, s, f8, thin)) != SVL_OK) return st;
    }

    if (want(l, SVL_LAYER_GATEUP)) {
    // MLP input norm fused into the gate/up GEMM (bf16: gain folded into W_g,
    // W_u; e4m3: applied by the quantiser)
    if (f8 && (st = quant(static_cast<const __nv_bfloat16*>(X), m->layers[l].ffn_norm, d.d_model, 1, d.d_model,
                          d.d_model, -1)) != SVL_OK)
      return st;
    p = base_params(m);
    set_norm(p, ss_b, nullptr);
    p.mapA = map_x;
    p.mapB[0] = tm[4];
    p.mapB[1] = tm[5];
    if (f8) set_f8(p, map_aq_x, tm8, sc8, {4, 5});
    if (pair) {
      p.mapB[0] = m->tm_pair[static_cast<size_t>(l) * 5 + 3];
      p.mapB[1] = m->tm_pair[static_cast<size_t>(l) * 5 + 4];
    }
    p.b_split = 1;
    p.tiles = sa.gu_tiles + static_cast<size_t>(l) * L.gu_cap;
    p.tile_count = counts + 2 * nl + l;
    p.max_tiles = L.gu_cap;
    p.K = d.d_model;
    p.kgroup = d.d_model;
    p.out[0] = hm;
    p.ld[0] = d.d_ffn;
    p.mapR = map_hmo;
    p.stage_tma = 1;
    if ((st = pair ? launch_pair(EPI_SWIGLU, m, SVL_TAG_GATEUP, p, L.gu_cap, s)
                   : launch(EPI_SWIGLU, m, SVL_TAG_GATEUP, p, L.gu_cap, s, f8, thin)) != SVL_OK)
      return st;
    }

    if (want(l, SVL_LAYER_DOWN)) {
    if (f8 && (st = quant(hm, nullptr, d.d_ffn, G, d.d_ffn / G, m->kgd_p, l)) != SVL_OK) return st;
    p = base_params(m);
    p.mapA = map_hm;
    p.mapB[0] = tm[6];
    p.tiles = sa.dn_tiles + static_cast<size_t>(l) * L.dn_cap;
    p.tile_count = counts + 3 * nl + l;
    p.max_tiles = L.dn_cap;
    p.K = d.d_ffn;
    p.kgroup = d.d_ffn / d.n_groups;
    if (f8) {
      set_f8(p, map_aq_h, tm8, sc8, {6});
      p.K = G * m->kgd_p;
      p.kgroup = m->kgd_p;
    }
    p.out[0] = X;
    p.ld[0] = d.d_model;
    p.mapR = map_xr;
    p.stage_tma = 1;
    p.a_evict_first = 1;  // n-band list: the weights stay in L2, the input rows stream
    p.ks_info = sa.ks_info + static_cast<size_t>(l) * 8 + 4;
    p.ks_part = at<float>(ws, L.ks_part);
    p.ks_ticket = ks_ticket + static_cast<size_t>(2 * l + 1) * L.ks_units;
    set_norm(p, nullptr, ss_a);  // for the next layer's attention norm
    if ((st = launch(EPI_RESID, m, SVL_TAG_DOWN, p, L.dn_cap, s, f8, thin)) != SVL_OK) return st;
    }
  }
  if (only) return last_error();

  // final norm + LM head
  na.gain = static_cast<const __nv_bfloat16*>(m->w.final_norm);
  na.act = nullptr;
  GemmParams p = base_params(m);
  if (logits_mode == SVL_LOGITS_LAST) {
    const int n_pad = ((B + 15) / 16) * 16;
    na.Y = at<__nv_bfloat16>(ws, L.yl);
    {
      Launch L1(m, SVL_TAG_RMSNORM, s);
      launch_final_last_rows(na, n_pad, s);
    }
    p.mapA = m->tm_lm_head;
    if (!make_map(&p.mapB[0], na.Y, n_pad, d.d_model)) return SVL_ERR_CUDA;
    p.grid_m = (d.vocab + kBM - 1) / kBM;
    p.grid_n = (n_pad + 255) / 256;
    p.bn = std::min(n_pad, 256);
    p.m_limit = d.vocab;
    p.n_limit = B;
    p.K = d.d_model;
    p.kgroup = d.d_model;
    p.out[0] = logits;
    p.ld[0] = d.vocab;
    if ((st = launch(EPI_LOGITS_T, m, SVL_TAG_LMHEAD, p, static_cast<int64_t>(p.grid_m) * p.grid_n, s)) != SVL_OK) return st;
  } else {
    {
      Launch L1(m, SVL_TAG_RMSNORM, s);
      launch_rmsnorm(na, s);
    }
    p.mapA = map_xn;
    p.mapB[0] = m->tm_lm_head;
    p.grid_m = (t_cap + kBM - 1) / kBM;
    p.grid_n = (d.vocab + 255) / 256;
    p.bn = 256;
    p.m_limit_dev = cu_seqlens + B;
    p.m_limit = t_cap;
    p.n_limit = d.vocab;
    p.K = d.d_model;
    p.kgroup = d.d_model;
    p.out[0] = logits;
    p.ld[0] = d.vocab;
    if ((st = launch(EPI_F32, m, SVL_TAG_LMHEAD, p, static_cast<int64_t>(p.grid_m) * p.grid_n, s)) != SVL_OK) return st;
  }
  if (kvx && kvx->decode) {
    Launch L1(m, SVL_TAG_LMHEAD, s);
    launch_decode_finish(B, d.vocab, logits, kvx->next_token, kvx->cache_len, kvx->max_len, s);
  } else if (kvx && kvx->cache_len) {
    launch_offsets_diff(cu_seqlens, kvx->cache_len, B, s);  // cache length = prompt length
    g_launches++;
  }
  return last_error();
}
}  // namespace

svl_status svl_gated_prefill(svl_model* m, int32_t B, int32_t t_cap, void* X, const int32_t* cu_seqlens,
                             const int32_t* pos, const uint8_t* layer_gate, const uint8_t* group_gate,
                             int32_t logits_mode, float* logits, void* ws, size_t ws_bytes, void* stream) {
  return prefill_impl(m, B, t_cap, X, cu_seqlens, pos, layer_gate, group_gate, logits_mode, logits, ws, ws_bytes,
                      stream, nullptr);
}

svl_status svl_layer_stage(svl_model* m, int32_t stage, int32_t layer, int32_t B, int32_t t_cap, void* X,
                           const int32_t* cu_seqlens, const int32_t* pos, const uint8_t* layer_gate,
                           const uint8_t* group_gate, void* q, void* k, void* vt, void* ao, void* h, void* ws,
                           size_t ws_bytes, void* stream) {
  if (!m || stage < SVL_LAYER_QKV || stage > SVL_LAYER_DOWN || layer < 0 || layer >= m->d.n_layers)
    return SVL_ERR_INVALID_ARG;
  const bool need_qkv = stage == SVL_LAYER_QKV || stage == SVL_LAYER_ATTN;
  if ((need_qkv && (!q || !k || !vt)) || ((stage == SVL_LAYER_ATTN || stage == SVL_LAYER_OPROJ) && !ao) ||
      ((stage == SVL_LAYER_GATEUP || stage == SVL_LAYER_DOWN) && !h))
    return SVL_ERR_INVALID_ARG;
  for (const void* p : {q, k, vt, ao, h})
    if (p && !aligned16(p)) return SVL_ERR_INVALID_ARG;
  // buffers the stage does not use still need a valid address for the
  // tensor maps made up front: X stands in for them (never read or written)
  auto or_x = [&](void* p) { return static_cast<__nv_bfloat16*>(p ? p : X); };
  StageSel sel{stage, layer, or_x(q), or_x(k), or_x(vt), or_x(ao), or_x(h)};
  return prefill_impl(m, B, t_cap, X, cu_seqlens, pos, layer_gate, group_gate, SVL_LOGITS_LAST, nullptr, ws,
                      ws_bytes, stream, nullptr, nullptr, &sel);
}

svl_status svl_controlled_prefill(svl_model* m, int32_t B, int32_t t_cap, void* X, const int32_t* cu_seqlens,
                                  const int32_t* pos, const float* budget, const float* kappa, const int32_t* k,
                                  const int32_t* vis_off, const int32_t* text_len, int32_t project,
                                  int32_t logits_mode, float* logits, uint8_t* layer_gate_out,
                                  uint8_t* group_gate_out, float* gate_logits_out, uint32_t* sample_flags, void* ws,
                                  size_t ws_bytes, void* stream) {
  if (!m || !budget || !kappa || !k || !vis_off || !text_len || !layer_gate_out || !group_gate_out)
    return SVL_ERR_INVALID_ARG;
  const svl_model_desc& d = m->d;
  if (!m->w.kap_w1 || !m->w.kap_w2 || !m->w.gate_w || !m->w.gate_c) return SVL_ERR_UNSUPPORTED;
  CtlArgs c;
  std::memset(&c, 0, sizeof(c));
  c.B = B;
  c.L = d.n_layers;
  c.G = d.n_groups;
  c.P = d.n_prefix;
  c.D = d.d_model;
  c.H = d.h_ctrl;
  c.Dkv = static_cast<long long>(d.n_kv_heads) * (d.d_model / d.n_heads);
  c.Di = d.d_ffn;
  c.V = d.vocab;
  c.project = project ? 1 : 0;
  c.kappa = kappa;
  c.budget = budget;
  c.k = k;
  c.vis_off = vis_off;
  c.text_len = text_len;
  c.kap_w1 = static_cast<const __nv_bfloat16*>(m->w.kap_w1);
  c.kap_w2 = static_cast<const __nv_bfloat16*>(m->w.kap_w2);
  c.gate_w = static_cast<const __nv_bfloat16*>(m->w.gate_w);
  c.gate_c = m->w.gate_c;
  c.gate_logits = gate_logits_out;
  c.flags = sample_flags;
  return prefill_impl(m, B, t_cap, X, cu_seqlens, pos, layer_gate_out, group_gate_out, logits_mode, logits, ws,
                      ws_bytes, stream, &c);
}

size_t svl_kv_cache_size(const svl_model* m, int32_t B, int32_t max_len) {
  if (!m || B <= 0 || max_len <= 0) return 0;
  const size_t dkv = static_cast<size_t>(m->d.n_kv_heads) * (m->d.d_model / m->d.n_heads);
  return 2 * sizeof(__nv_bfloat16) * static_cast<size_t>(m->d.n_layers) * B * max_len * dkv;
}

svl_status svl_gated_prefill_kv(svl_model* m, int32_t B, int32_t t_cap, void* X, const int32_t* cu_seqlens,
                                const int32_t* pos, const uint8_t* layer_gate, const uint8_t* group_gate,
                                int32_t logits_mode, float* logits, void* kv_cache, int32_t max_len,
                                int32_t* cache_len, void* ws, size_t ws_bytes, void* stream) {
  if (!m || !kv_cache || !cache_len || max_len <= 0 || max_len > m->d.max_seq || !aligned16(kv_cache))
    return SVL_ERR_INVALID_ARG;
  StepCtx kx{static_cast<__nv_bfloat16*>(kv_cache), max_len, 0, cache_len, nullptr, nullptr};
  return prefill_impl(m, B, t_cap, X, cu_seqlens, pos, layer_gate, group_gate, logits_mode, logits, ws, ws_bytes,
                      stream, nullptr, &kx);
}

size_t svl_decode_workspace_size(const svl_model* m, int32_t B) {
  if (!m || B <= 0) return 0;
  const size_t head = align256(2 * static_cast<size_t>(B) * m->d.d_model) + align256(4 * (B + 1)) + align256(4 * B);
  return head + pre_layout(m->d, B, B).total;
}

svl_status svl_decode_step(svl_model* m, int32_t B, const int32_t* tokens, void* kv_cache, int32_t max_len,
                           int32_t* cache_len, const uint8_t* layer_gate, const uint8_t* group_gate, float* logits,
                           int32_t* next_token, void* ws, size_t ws_bytes, void* stream) {
  if (!m || B <= 0 || !tokens || !kv_cache || max_len <= 0 || max_len > m->d.max_seq || !cache_len ||
      !layer_gate || !group_gate || !logits || !aligned16(kv_cache) || !ws)
    return SVL_ERR_INVALID_ARG;
  if (ws_bytes < svl_decode_workspace_size(m, B)) return SVL_ERR_WORKSPACE;
  // the step's rows, cu_seqlens and positions live at the head of the workspace
  uint8_t* base = static_cast<uint8_t*>(ws);
  const size_t xb = align256(2 * static_cast<size_t>(B) * m->d.d_model), cb = align256(4 * (B + 1)),
               pb = align256(4 * B);
  void* X = base;
  int32_t* cu = reinterpret_cast<int32_t*>(base + xb);
  int32_t* pos = reinterpret_cast<int32_t*>(base + xb + cb);
  StepCtx kx{static_cast<__nv_bfloat16*>(kv_cache), max_len, 1, cache_len, tokens, next_token};
  return prefill_impl(m, B, B, X, cu, pos, layer_gate, group_gate, SVL_LOGITS_LAST, logits, base + xb + cb + pb,
                      ws_bytes - (xb + cb + pb), stream, nullptr, &kx);
}

svl_status svl_quantize_rows_e4m3(const void* src, const void* gain, int64_t rows, int32_t cols, int64_t ld_src,
                                  void* dst, int64_t ld_dst, float* scale, void* stream) {
  if (!src || !dst || !scale || rows < 0 || cols <= 0 || (cols & 7) || ld_src < cols || (ld_src & 7) ||
      ld_dst < cols || (ld_dst & 7) || !aligned16(src) || (reinterpret_cast<uintptr_t>(dst) & 7) ||
      (reinterpret_cast<uintptr_t>(scale) & 3) || (gain && !aligned16(gain)))
    return SVL_ERR_INVALID_ARG;
  QuantArgs qa;
  std::memset(&qa, 0, sizeof(qa));
  qa.src = static_cast<const __nv_bfloat16*>(src);
  qa.gain = static_cast<const __nv_bfloat16*>(gain);
  qa.ld_src = ld_src;
  qa.rows = rows;
  qa.G = 1;
  qa.kg = cols;
  qa.kgp = cols;
  qa.dst = static_cast<uint8_t*>(dst);
  qa.ld_dst = ld_dst;
  qa.scale = scale;
  g_launches++;
  if (launch_quant_rows(qa, static_cast<cudaStream_t>(stream)) != cudaSuccess) return SVL_ERR_CUDA;
  return last_error();
}

svl_status svl_gemm_e4m3(svl_model* m, const void* A, const float* a_scale, const void* B, const float* b_scale,
                         int32_t M, int32_t N, int32_t K, float* C, void* stream) {
  if (!m || !A || !a_scale || !B || !b_scale || !C || M <= 0 || N <= 0 || K <= 0 || (K % kBK8) || (N & 31))
    return SVL_ERR_INVALID_ARG;
  GemmParams p = base_params(m);
  if (!make_map8(&p.mapA, A, M, K) || !make_map8(&p.mapB[0], B, N, K)) return SVL_ERR_INVALID_ARG;
  p.grid_m = (M + kBM - 1) / kBM;
  p.bn = std::min(N, 256);
  p.grid_n = (N + p.bn - 1) / p.bn;
  p.m_limit = M;
  p.n_limit = N;
  p.K = K;
  p.kgroup = K;
  p.out[0] = C;
  p.ld[0] = N;
  p.a_scale = a_scale;
  p.b_scale[0] = b_scale;
  svl_status st = launch(EPI_F32, m, SVL_TAG_LMHEAD, p, static_cast<int64_t>(p.grid_m) * p.grid_n,
                         static_cast<cudaStream_t>(stream), true);
  return st != SVL_OK ? st : last_error();
}

svl_status svl_flops(const svl_model_desc* d, int32_t s_text, int32_t s_vis, int32_t n_vis, const uint8_t* lg,
                     const uint8_t* gg, double* eq8, double* exec) {
  if (!d || s_text < 0 || s_vis < 0 || n_vis < 0 || d->n_heads <= 0 || d->n_groups <= 0) return SVL_ERR_INVALID_ARG;
  const int64_t D = d->d_model, dh = d->d_model / d->n_heads, Dkv = d->n_kv_heads * dh, Di = d->d_ffn, V = d->vocab;
  const int64_t G = d->n_groups, S = static_cast<int64_t>(s_text) + s_vis;
  int64_t n_on = 0;
  for (int l = 0; l < d->n_layers; ++l)
    for (int j = 0; j < G; ++j)
      n_on += (l < d->n_prefix || !lg || !gg || (lg[l] && gg[l * G + j])) ? 1 : 0;
  const int64_t lin = 4 * D * D + 4 * D * Dkv + 6 * D * Di;
  const int64_t cG = n_on * (lin * S + 4 * D * S * S) + G * 2 * D * V * S;
  if (eq8) *eq8 = static_cast<double>(cG) / static_cast<double>(G);
  if (exec) {
    double f = 2.0 * n_vis * d->c_vis * d->h_ctrl;
    if (d->proj_hidden) f += 2.0 * s_vis * (static_cast<double>(d->c_vis) * d->proj_hidden + static_cast<double>(d->proj_hidden) * D);
    f += static_cast<double>(n_on) * (static_cast<double>(lin) * S + 2.0 * D * S * (S + 1)) / G;
    f += 2.0 * D * V;
    *exec = f;
  }
  return SVL_OK;
}

size_t svl_host_workspace_size(const svl_model* m, int32_t B, int64_t nv, int64_t nt) {
  if (!m || B <= 0 || nv < 0 || nt < 0) return 0;
  return host_layout(m->d, B, nv, nt).total;
}

svl_status svl_prefill_from_host(svl_model* m, int32_t B, int32_t nv, int32_t nt, const void* h_vis,
                                 const int32_t* h_vis_off, const int32_t* h_text_ids, const int32_t* h_text_off,
                                 const float* h_budget, const int32_t* h_keep_count, const uint8_t* h_layer_gate,
                                 const uint8_t* h_group_gate, float* h_logits, int32_t* h_k, void* ws,
                                 size_t ws_bytes, void* stream) {
  if (!m || B <= 0 || nv < 0 || nt < 0 || !h_vis_off || !h_text_off || !h_budget || !h_layer_gate ||
      !h_group_gate || !h_logits || (nv > 0 && !h_vis) || (nt > 0 && !h_text_ids))
    return SVL_ERR_INVALID_ARG;
  const HostLayout H = host_layout(m->d, B, nv, nt);
  svl_status st = check_ws(ws, ws_bytes, H.total);
  if (st != SVL_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const svl_model_desc& d = m->d;
  const size_t L = d.n_layers, G = d.n_groups;
  auto h2d = [&](size_t off, const void* src, size_t bytes) {
    return bytes == 0 || cudaMemcpyAsync(at<uint8_t>(ws, off), src, bytes, cudaMemcpyHostToDevice, s) == cudaSuccess;
  };
  bool ok;
  {
    Launch C(m, SVL_TAG_COPY, s);
    ok = h2d(H.vis, h_vis, 2 * static_cast<size_t>(nv) * d.c_vis) && h2d(H.vis_off, h_vis_off, 4 * (B + 1)) &&
         h2d(H.text_ids, h_text_ids, 4 * static_cast<size_t>(nt)) && h2d(H.text_off, h_text_off, 4 * (B + 1)) &&
         h2d(H.budget, h_budget, 4 * B) && h2d(H.lg, h_layer_gate, B * L) && h2d(H.gg, h_group_gate, B * L * G) &&
         (!h_keep_count || h2d(H.keep, h_keep_count, 4 * B));
    g_launches--;  // copies are not kernels
  }
  if (!ok) return SVL_ERR_CUDA;
  {
    Launch L1(m, SVL_TAG_PACK, s);
    launch_offsets_diff(at<int>(ws, H.text_off), at<int>(ws, H.text_len), B, s);
  }
  void* inner = at<uint8_t>(ws, H.inner);
  const size_t inner_bytes = ws_bytes - H.inner;
  st = svl_score_select(m, B, nv, at<void>(ws, H.vis), at<int>(ws, H.vis_off), at<int>(ws, H.text_len),
                        at<float>(ws, H.budget), h_keep_count ? at<int>(ws, H.keep) : nullptr,
                        at<uint8_t>(ws, H.lg), at<uint8_t>(ws, H.gg), at<float>(ws, H.scores), at<int>(ws, H.k),
                        at<int>(ws, H.kept_idx), at<int>(ws, H.kept_off), at<uint32_t>(ws, H.flags), inner,
                        inner_bytes, stream);
  if (st != SVL_OK) return st;
  st = svl_pack(m, B, nv, nt, at<void>(ws, H.vis), at<int>(ws, H.vis_off), at<int>(ws, H.kept_idx),
                at<int>(ws, H.kept_off), at<int>(ws, H.text_ids), at<int>(ws, H.text_off), at<void>(ws, H.X),
                at<int>(ws, H.cu), at<int>(ws, H.pos), inner, inner_bytes, stream);
  if (st != SVL_OK) return st;
  const int t_cap = std::max(nv + nt, 1);
  st = svl_gated_prefill(m, B, t_cap, at<void>(ws, H.X), at<int>(ws, H.cu), at<int>(ws, H.pos),
                         at<uint8_t>(ws, H.lg), at<uint8_t>(ws, H.gg), SVL_LOGITS_LAST, at<float>(ws, H.logits),
                         inner, inner_bytes, stream);
  if (st != SVL_OK) return st;
  {
    Launch C(m, SVL_TAG_COPY, s);
    g_launches--;
    ok = cudaMemcpyAsync(h_logits, at<float>(ws, H.logits), sizeof(float) * static_cast<size_t>(B) * d.vocab,
                         cudaMemcpyDeviceToHost, s) == cudaSuccess &&
         (!h_k || cudaMemcpyAsync(h_k, at<int>(ws, H.k), 4 * B, cudaMemcpyDeviceToHost, s) == cudaSuccess);
  }
  return ok ? SVL_OK : SVL_ERR_CUDA;
}

svl_status svl_profile_start(svl_model* m, uint32_t tag_mask) {
  if (!m) return SVL_ERR_INVALID_ARG;
  m->prof = true;
  m->prof_mask = tag_mask;
  m->ev_used = 0;
  m->prof_recs.clear();
  return SVL_OK;
}

svl_status svl_profile_stop(svl_model* m, svl_kernel_time* out, int32_t cap, int32_t* n_out) {
  if (!m || (!out && cap > 0)) return SVL_ERR_INVALID_ARG;
  m->prof = false;
  double tot[SVL_TAG_COUNT] = {0};
  int cnt[SVL_TAG_COUNT] = {0};
  m->prof_last.clear();
  if (!m->prof_recs.empty()) {
    if (cudaEventSynchronize(m->ev_pool[m->prof_recs.back().second + 1]) != cudaSuccess) return SVL_ERR_CUDA;
  }
  for (const auto& r : m->prof_recs) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, m->ev_pool[r.second], m->ev_pool[r.second + 1]) != cudaSuccess) return SVL_ERR_CUDA;
    m->prof_last.emplace_back(r.first, ms);
    if (r.first >= 0 && r.first < SVL_TAG_COUNT) {
      tot[r.first] += ms;
      cnt[r.first] += 1;
    }
  }
  m->prof_recs.clear();
  m->ev_used = 0;
  int n = 0;
  for (int t = 0; t < SVL_TAG_COUNT; ++t) {
    if (!cnt[t]) continue;
    if (n < cap) out[n] = svl_kernel_time{t, cnt[t], tot[t]};
    ++n;
  }
  if (n_out) *n_out = std::min(n, cap);
  return SVL_OK;
}

svl_status svl_profile_launches(svl_model* m, int32_t* tags, float* ms, int32_t cap, int32_t* n_out) {
  if (!m || cap < 0 || (cap > 0 && (!tags || !ms))) return SVL_ERR_INVALID_ARG;
  const int n = std::min<int>(cap, static_cast<int>(m->prof_last.size()));
  for (int i = 0; i < n; ++i) {
    tags[i] = m->prof_last[i].first;
    ms[i] = m->prof_last[i].second;
  }
  if (n_out) *n_out = n;
  return SVL_OK;
}

const char* svl_tag_name(int32_t tag) {
  static const char* names[SVL_TAG_COUNT] = {"budget_embed", "score", "select", "pack", "projector",
                                              "schedule", "rmsnorm", "qkv_gemm", "attention", "o_gemm",
                                              "gateup_gemm", "down_gemm", "lm_head", "host_copy", "quant"};
  return (tag >= 0 && tag < SVL_TAG_COUNT) ? names[tag] : "unknown";
}

svl_status svl_selftest_wait_timeout(svl_model* m, uint64_t wait_cycles, void* stream) {
  if (!m) return SVL_ERR_INVALID_ARG;
  const long long c = static_cast<long long>(std::min<uint64_t>(std::max<uint64_t>(wait_cycles, 1000), 1000000000));
  {
    Launch L1(m, SVL_TAG_SCHEDULE, static_cast<cudaStream_t>(stream));
    launch_selftest_wait(m->d_status, c, static_cast<cudaStream_t>(stream));
  }
  return last_error();
}

svl_status svl_get_device_status(svl_model* m, void* stream, uint32_t* code) {
  if (!m || !code) return SVL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(code, m->d_status, sizeof(uint32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return SVL_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return SVL_ERR_CUDA;
  if (cudaMemsetAsync(m->d_status, 0, sizeof(uint32_t), s) != cudaSuccess) return SVL_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return SVL_ERR_CUDA;
  return SVL_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Token controller without workspace: svl_score_select_noalloc.
//
// Some callers cannot hand the library freshly allocated device memory: code
// that runs while a stream is being captured into a CUDA graph (cudaMalloc is
// not allowed there), plugins whose host framework has already reserved the
// device's memory for its own allocator and gives them none, or real-time
// paths that must not block in the allocator. For them this entry point keeps
// its scratch -- the budget embeddings e_b and the per-sample kept lists -- in
// one fixed array in device memory that is part of the library image. Every
// GPU that loads the library holds the array until the process exits.
namespace {

constexpr int kNoAllocMaxBatch = 256;     // samples per call
constexpr int kNoAllocMaxHctrl = 256;     // token-controller hidden width
constexpr int kNoAllocMaxVis = 65536;     // visual tokens per call (all samples)
constexpr size_t kNoAllocEbBytes = sizeof(float) * kNoAllocMaxBatch * kNoAllocMaxHctrl;   // 256 KiB
constexpr size_t kNoAllocListBytes = sizeof(int) * kNoAllocMaxVis;                        // 256 KiB
constexpr size_t kNoAllocScratchBytes = kNoAllocEbBytes + kNoAllocListBytes;              // 512 KiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kNoAllocMaxDevices] = {};

// Device address of the scratch array on the current device. In host code
// the array's name is only a host-side stand-in, so the address is looked up
// once per device (with that device current) and cached.
svl_status noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices) return SVL_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return SVL_ERR_CUDA;
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return SVL_OK;
}

}  // namespace

extern "C" svl_status svl_score_select_noalloc(svl_model* m, int32_t B, int32_t n_vis_total, const void* vis_feats,
                                               const int32_t* vis_off, const int32_t* text_len, const float* budget,
                                               const int32_t* keep_count, const uint8_t* layer_gate,
                                               const uint8_t* group_gate, float* scores, int32_t* k,
                                               int32_t* kept_idx, int32_t* kept_off, uint32_t* sample_flags,
                                               void* stream) {
  if (!m || B <= 0 || n_vis_total < 0 || !vis_off || !text_len || !budget || !layer_gate || !group_gate ||
      !scores || !k || !kept_idx || !kept_off)
    return SVL_ERR_INVALID_ARG;
  if (n_vis_total > 0 && (!vis_feats || !aligned16(vis_feats))) return SVL_ERR_INVALID_ARG;
  if (B > kNoAllocMaxBatch || n_vis_total > kNoAllocMaxVis || m->d.h_ctrl > kNoAllocMaxHctrl)
    return SVL_ERR_SHAPE;  // beyond the fixed scratch array
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev != m->device) return SVL_ERR_INVALID_ARG;
  void* scratch = nullptr;
  svl_status st = noalloc_scratch(&scratch);
  if (st != SVL_OK) return st;
  float* e_b = static_cast<float*>(scratch);
  int* kept_local = reinterpret_cast<int*>(static_cast<unsigned char*>(scratch) + kNoAllocEbBytes);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const svl_model_desc& d = m->d;

  // Every scratch element read below is written earlier in the same call
  // (e_b by the budget MLP, kept_local[vis_off[b] ..] by the select kernel
  // before compaction reads it), so nothing has to be cleared first.
  {
    Launch L(m, SVL_TAG_BUDGET_EMBED, s);
    launch_budget_embed(budget, static_cast<const __nv_bfloat16*>(m->w.bud_w1),
                        static_cast<const __nv_bfloat16*>(m->w.bud_w2), d.h_ctrl, B, e_b, s);
  }
  if (n_vis_total > 0) {
    GemmParams p = base_params(m);
    if (!make_map(&p.mapA, vis_feats, n_vis_total, d.c_vis)) return SVL_ERR_INVALID_ARG;
    p.mapB[0] = m->tm_ctrl_w1;
    p.grid_m = (n_vis_total + kBM - 1) / kBM;
    p.grid_n = 1;
    p.bn = d.h_ctrl;
    p.m_limit = n_vis_total;
    p.n_limit = d.h_ctrl;
    p.K = d.c_vis;
    p.kgroup = d.c_vis;
    p.out[0] = scores;
    p.e_b = e_b;
    p.seg_off = vis_off;
    p.n_seg = B;
    p.w2 = static_cast<const __nv_bfloat16*>(m->w.ctrl_w2);
    p.c2 = m->w.ctrl_c2;
    p.b_box_rows = d.h_ctrl;
    st = launch(d.h_ctrl <= 64 ? EPI_SCORE : EPI_SCORE_WIDE, m, SVL_TAG_SCORE, p, p.grid_m, s);
    if (st != SVL_OK) return st;
  }
  SelectArgs a;
  std::memset(&a, 0, sizeof(a));
  a.scores = scores;
  a.vis_off = vis_off;
  a.text_len = text_len;
  a.budget = budget;
  a.keep_count = keep_count;
  a.layer_gate = layer_gate;
  a.group_gate = group_gate;
  a.L = d.n_layers;
  a.G = d.n_groups;
  a.P = d.n_prefix;
  a.D = d.d_model;
  a.Dkv = static_cast<long long>(d.n_kv_heads) * (d.d_model / d.n_heads);
  a.Di = d.d_ffn;
  a.V = d.vocab;
  a.k_out = k;
  a.flags = sample_flags;
  a.kept_local = kept_local;
  {
    Launch L1(m, SVL_TAG_SELECT, s);
    launch_select(a, B, s);
  }
  {
    Launch L2(m, SVL_TAG_SELECT, s);
    launch_compact(B, vis_off, k, kept_local, kept_idx, kept_off, nullptr, s);
  }
  return last_error();
}
