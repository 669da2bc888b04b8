/*
 * svl.h -- C ABI of the GB300 (sm_103a) budget-conditioned gated prefill.
 *
 * The library implements the inference hot path of SmartVL ("Look Less, Think
 * Faster: Joint Token-Compute Adaptation for Multimodal LLMs", arXiv
 * 2607.20357): the vision-side token controller that scores visual tokens
 * under a budget and keeps the top k of each sample (Sec. 3.1, Sec. 3.3
 * "Inference"), the packing of kept visual tokens and text tokens into one
 * variable-length batch (Sec. 3.1, contiguous RoPE), and the LLM decoder
 * forward under per-sample layer / head-group gates (Sec. 3.2) where gated-off
 * work is never issued.
 *
 * Conventions shared by every call below.
 *  - All tensor arguments are DEVICE pointers owned by the caller, unless the
 *    name says host. bf16 tensors are IEEE bfloat16, row-major, contiguous.
 *  - Calls that take a stream are asynchronous on it. Apart from
 *    svl_get_device_status and svl_profile_stop, the library never
 *    synchronises, and only svl_prefill_from_host copies results to the host.
 *    Counts that depend on data (k, sequence lengths, tile lists) stay on the
 *    device.
 *  - The returned status reports argument and shape errors found on the host;
 *    in that case nothing was launched. Data-dependent errors (a non-finite
 *    token logit, a device wait that ran out of time) are OR-ed into the
 *    model's device status word, read with svl_get_device_status().
 *  - `workspace` is caller-allocated device memory of at least
 *    svl_workspace_size() bytes, 256-byte aligned. Calls that share a
 *    workspace must be ordered on one stream.
 *  - Gates are bytes, 0 = off, anything else = on. For layers l < n_prefix
 *    the gates are ignored and every group runs (Sec. 3.2 prefix layers).
 *  - The GEMM and attention kernels are persistent (one CTA per SM) and the
 *    shares of a GEMM's K-split tail wait for each other inside one launch.
 *    Run the calls of one GPU on one stream (or ordered streams): two of them
 *    running concurrently can keep each other's CTAs off the SMs until a
 *    bounded wait gives up (SVL_DEV_TIMEOUT in the status word).
 *
 * Beyond the three calls of the path: svl_score_select_paper (the paper's own
 * inference rule, Sec. 3.1 and Sec. 3.3), svl_pack_controlled and
 * svl_controlled_prefill (the LLM-side compute controller, Sec. 3.2, Eq. 7),
 * svl_gated_prefill_kv and svl_decode_step (gated decode with a KV cache,
 * which the paper leaves open, Sec. 5), gemm_format = SVL_GEMM_E4M3 with
 * svl_quantize_rows_e4m3 and svl_gemm_e4m3 (FP8 gated projections; Sec. 5
 * calls quantisation orthogonal to the method), svl_prefill_from_host (the
 * path from host buffers), svl_flops (Eq. 8 on the host) and the profiling and
 * self-test calls.
 */
#ifndef SVL_H
#define SVL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum svl_status {
  SVL_OK = 0,
  SVL_ERR_INVALID_ARG = 1,   /* null pointer, negative size, bad enum value */
  SVL_ERR_SHAPE = 2,         /* sizes inconsistent with the model or the workspace */
  SVL_ERR_UNSUPPORTED = 3,   /* dims the kernels do not support (see svl_model_create) */
  SVL_ERR_CUDA = 4,          /* a CUDA runtime call failed */
  SVL_ERR_NONFINITE = 5,     /* device status bit: a token logit was NaN or infinite */
  SVL_ERR_TIMEOUT = 6,       /* device status bit: a bounded device wait gave up */
  SVL_ERR_WORKSPACE = 7      /* workspace null, too small or misaligned */
} svl_status;

/* Device status word bits (svl_get_device_status). */
#define SVL_DEV_NONFINITE 0x1u
#define SVL_DEV_TIMEOUT 0x2u
#define SVL_DEV_BAD_INDEX 0x4u

/* Per-sample flag bits written by svl_score_select. */
#define SVL_FLAG_OVER_BUDGET 0x1u /* even zero visual tokens exceed b * C_full */
#define SVL_FLAG_GROUPS_DROPPED 0x2u /* paper rule: the budget projection switched head groups off */

/* Model dimensions.  Notation of Sec. 3: L layers, width D, A heads, FFN
 * width D_int, vocabulary V, G head groups, P prefix layers; C_v is the
 * vision feature width; H the token-controller hidden width.
 * Supported: D = A * d_head with d_head in {64, 128}; A % G == 0 and
 * A_kv % G == 0 (each group owns whole KV heads); (D_int / G) % 64 == 0;
 * (A / G) * d_head % 64 == 0; D a multiple of 128; C_v, proj_hidden
 * multiples of 64;
 * H in {16, 32, ..., 128}; proj_hidden == 0 requires C_v == D.
 *
 * gemm_format selects the operand type of the four gated projections of
 * every decoder layer (QKV, O, gate/up, down): SVL_GEMM_BF16, or
 * SVL_GEMM_E4M3 -- FP8 weights, which the paper calls orthogonal to its
 * method (Sec. 5). With e4m3, svl_model_create quantises each weight output
 * channel (row of W as given) to e4m3 with the scale amax / 448; each
 * activation row feeding those GEMMs -- RMSNorm(X) * gain for QKV and
 * gate/up, the attention output for O, the SwiGLU output for down -- is
 * quantised the same way on the fly (svl_quantize_rows_e4m3 is the
 * definition), and the fp32 accumulator of the code products is scaled by
 * both rows' scales. The projector, token controller and LM head stay
 * bf16. */
#define SVL_GEMM_BF16 0
#define SVL_GEMM_E4M3 1
typedef struct svl_model_desc {
  int32_t n_layers;     /* L */
  int32_t d_model;      /* D */
  int32_t n_heads;      /* A */
  int32_t n_kv_heads;   /* A_kv (GQA when < A) */
  int32_t d_ffn;        /* D_int (SwiGLU) */
  int32_t vocab;        /* V */
  int32_t n_groups;     /* G */
  int32_t n_prefix;     /* P */
  int32_t c_vis;        /* C_v */
  int32_t h_ctrl;       /* H */
  int32_t proj_hidden;  /* LLaVA projector hidden width; 0 = identity */
  float rms_eps;
  float rope_theta;
  int32_t max_seq;      /* longest per-sample sequence the model will see */
  int32_t gemm_format;  /* SVL_GEMM_BF16 or SVL_GEMM_E4M3 (gated projections) */
} svl_model_desc;

/* One decoder layer's weights: device bf16, nn.Linear layout [out, in]. */
typedef struct svl_layer_weights {
  const void* wq;         /* [A*d_head, D] */
  const void* wk;         /* [A_kv*d_head, D] */
  const void* wv;         /* [A_kv*d_head, D] */
  const void* wo;         /* [D, A*d_head] */
  const void* wg;         /* [D_int, D] */
  const void* wu;         /* [D_int, D] */
  const void* wd;         /* [D, D_int] */
  const void* attn_norm;  /* [D] RMSNorm gain */
  const void* ffn_norm;   /* [D] */
} svl_layer_weights;

/* All weights: device bf16 unless noted, 16-byte aligned. The model keeps
 * these pointers (it does not copy them): the caller keeps the memory alive
 * until svl_model_destroy(). One exception: RMSNorm is computed inside the
 * GEMMs that follow it, so a layer whose attn_norm (ffn_norm) gains are not
 * all exactly 1 gets model-owned copies of W_q, W_k, W_v (W_g, W_u) with the
 * gains folded into their columns, made once by svl_model_create. */
typedef struct svl_weights {
  const void* ctrl_w1;    /* [H, C_v]  token scorer, first layer */
  const void* ctrl_w2;    /* [H]       token scorer, output weights */
  float ctrl_c2;          /*           token scorer, output bias (host value) */
  const void* bud_w1;     /* [H, H]    budget MLP (Eq. 5) */
  const void* bud_w2;     /* [H, H] */
  const void* proj_w1;    /* [proj_hidden, C_v] or NULL */
  const void* proj_w2;    /* [D, proj_hidden] or NULL */
  const void* embed;      /* [V, D] token embedding */
  const void* final_norm; /* [D] */
  const void* lm_head;    /* [V, D] */
  const svl_layer_weights* layers; /* HOST array of n_layers entries */
  /* LLM-side compute controller (Sec. 3.2), used only by
   * svl_pack_controlled / svl_controlled_prefill; may be NULL otherwise. */
  const void* llm_bud_w1; /* [H, H]  budget-token MLP: e = W2 SiLU(W1 PE(b)), Eq. 5 encoding */
  const void* llm_bud_w2; /* [D, H] */
  const void* kap_w1;     /* [H, H]  token-count MLP of Eq. 7: W2 SiLU(W1 PE(kappa)) */
  const void* kap_w2;     /* [D, H] */
  const void* gate_w;     /* [(L - P) * G, D] gate head W_h (rows: layer P.., group) */
  const float* gate_c;    /* [(L - P) * G] gate head bias c_h, float32 */
} svl_weights;

typedef struct svl_model svl_model;

/* Creates a model on the current CUDA device: validates dims, records the
 * weight pointers, allocates the device status word and the RoPE cos/sin
 * table (max_seq x d_head/2 float2, computed in double precision).
 * Returns SVL_ERR_UNSUPPORTED for dims outside the list above.
 * With SVL_PAIR_GEMM=1 in the environment, a bf16 model runs its QKV and
 * gate/up GEMMs on clusters of two CTAs (256-row tiles, tcgen05
 * cta_group::2); the results meet the same bars, and the default
 * single-CTA kernel is as fast on GB300. */
svl_status svl_model_create(const svl_model_desc* desc, const svl_weights* weights, svl_model** out);
void svl_model_destroy(svl_model* model);

/* Bytes of workspace for batches of up to `max_batch` samples with at most
 * `max_vis_total` visual and `max_text_total` text tokens in total. */
size_t svl_workspace_size(const svl_model* model, int32_t max_batch, int64_t max_vis_total,
                          int64_t max_text_total);

#define SVL_STAGE_SELECT 1u  /* svl_score_select */
#define SVL_STAGE_PACK 2u    /* svl_pack */
#define SVL_STAGE_PREFILL 4u /* svl_gated_prefill */
/* Workspace bytes for only the stages in `stages` (a caller that only runs
 * the token controller needs far less than svl_workspace_size()). */
size_t svl_workspace_size_for(const svl_model* model, uint32_t stages, int32_t max_batch, int64_t max_vis_total,
                              int64_t max_text_total);

/* (1) Token controller (Sec. 3.1; Sec. 3.3 "Inference"; Eq. 5; Eq. 8).
 *  Scores every visual token, z_i = w2 . SiLU(W1 x_i + e_b) + c2, with the
 *  budget embedding e_b = W_b2 SiLU(W_b1 PE(b)); derives k_b as the largest
 *  count whose Eq. 8 cost (with the sample's gates) stays within b * C_full,
 *  or min(keep_count[b], N_b) when keep_count[b] >= 0; keeps the k_b highest
 *  logits (equal logits: lower index first) and writes their indices in
 *  ascending order, compacted over the batch.
 *   vis_feats   [n_vis_total, C_v] bf16; sample b owns rows vis_off[b]..vis_off[b+1)
 *   vis_off     [B+1] int32, vis_off[0] = 0, vis_off[B] = n_vis_total
 *   text_len    [B] int32 text tokens per sample (S_text)
 *   budget      [B] float32 b in (0, 1]
 *   keep_count  [B] int32 or NULL (NULL / negative: derive from the budget)
 *   layer_gate  [B, L] uint8; group_gate [B, L, G] uint8
 *  Outputs: scores [n_vis_total] float32; k [B] int32; kept_idx
 *  [n_vis_total] int32 (first sum(k) entries valid; indices are local to the
 *  sample); kept_off [B+1] int32; sample_flags [B] uint32. */
svl_status svl_score_select(svl_model* model, int32_t B, int32_t n_vis_total,
                            const void* vis_feats, const int32_t* vis_off, const int32_t* text_len,
                            const float* budget, const int32_t* keep_count,
                            const uint8_t* layer_gate, const uint8_t* group_gate,
                            float* scores, int32_t* k, int32_t* kept_idx, int32_t* kept_off,
                            uint32_t* sample_flags, void* workspace, size_t workspace_bytes,
                            void* stream);

/* The paper's own inference rule for the token controller (Sec. 3.1 and
 * Sec. 3.3 "Inference"), with the LLM-side gates given as the compute
 * controller's pre-threshold logits instead of 0/1 masks:
 *   - a visual token survives if sigma(z_i) > 0.5, i.e. z_i > 0;
 *   - group j of layer l runs if l < P or gate_logits[b, l, j] > 0;
 *   - budget projection against b * C_full (Eq. 2, Eq. 8): the kept count is
 *     k = min(#{z_i > 0}, the largest count within the budget for these
 *     gates), the lowest logits going first (ties: lower index);
 *   - if even k = 0 exceeds the budget, the fewest active groups of layers
 *     l >= P that bring the text-only cost within it are switched off, in
 *     increasing order of their logit (equal logits: lower l * G + j first);
 *     sample_flags gets SVL_FLAG_GROUPS_DROPPED, and also
 *     SVL_FLAG_OVER_BUDGET if the prefix layers alone exceed the budget
 *     (every other group is then off).
 * keep_count >= 0 overrides k as in svl_score_select (no projection).
 * Arguments as svl_score_select, except:
 *   gate_logits     [B, L, G] float32, device
 *   layer_gate_out  [B, L] uint8, device: 1 where any group of the layer runs
 *   group_gate_out  [B, L, G] uint8, device: the projected gates
 * The two gate outputs are what svl_gated_prefill takes. The comparison
 * z_i > 0 is made on the float32 logits written to `scores`. Workspace:
 * svl_workspace_size_for(..., SVL_STAGE_SELECT, ...). Errors: as
 * svl_score_select. */
svl_status svl_score_select_paper(svl_model* model, int32_t B, int32_t n_vis_total, const void* vis_feats,
                                  const int32_t* vis_off, const int32_t* text_len, const float* budget,
                                  const int32_t* keep_count, const float* gate_logits, float* scores,
                                  int32_t* k, int32_t* kept_idx, int32_t* kept_off, uint32_t* sample_flags,
                                  uint8_t* layer_gate_out, uint8_t* group_gate_out, float* kappa_out,
                                  void* workspace, size_t workspace_bytes, void* stream);
/* With gate_logits == NULL the gates are not known yet (the compute
 * controller decides them after the prefix layers, svl_controlled_prefill):
 * k = #{z_i > 0} (keep_count >= 0 overrides), no budget projection here, the
 * gate outputs may be NULL and are not written. kappa_out [B] (device, or
 * NULL) receives the token survival rate kappa = sum_i sigma(z_i) / N_b of
 * Sec. 3.2 (0 for N_b = 0), in both modes. */

/* Packs like svl_pack and appends to each sample its budget token (Sec. 3.2:
 * e_b = MLP_LLM(PE(b)) with the Eq. 5 encoding, weights llm_bud_w1/w2) as its
 * last row, position S_b. X, pos: room for n_vis_total + n_text_total + B
 * rows. Errors: as svl_pack; SVL_ERR_UNSUPPORTED without the controller
 * weights. */
svl_status svl_pack_controlled(svl_model* model, int32_t B, int32_t n_vis_total, int32_t n_text_total,
                               const void* vis_feats, const int32_t* vis_off, const int32_t* kept_idx,
                               const int32_t* kept_off, const int32_t* text_ids, const int32_t* text_off,
                               const float* budget, void* X, int32_t* cu_seqlens, int32_t* pos, void* workspace,
                               size_t workspace_bytes, void* stream);

/* The gated prefill with the LLM-side compute controller in the loop
 * (Sec. 3.2, Eq. 7): over a batch packed by svl_pack_controlled, the P
 * prefix layers run at full capacity; then, per sample, the budget token's
 * state h plus W_k2 SiLU(W_k1 PE(kappa)) feeds the linear gate head, group j
 * of layer l >= P runs if its logit is > 0, and with `project` != 0 and
 * b < 1 the fewest active groups (lowest logit first; equal logits: lower
 * l * G + j first) are switched off until Eq. 8 at S = S_text + k fits
 * b * C_full (Sec. 3.3; the token count is already committed). The device
 * schedule of the remaining layers is rebuilt from these gates with no host
 * round trip, and the logits come from each sample's last row (the budget
 * token, which the answer follows).
 *   budget, kappa   [B] float32, device (kappa from svl_score_select_paper)
 *   k, text_len     [B] int32, device: kept visual tokens, text tokens
 *   vis_off         [B+1] int32, device: visual tokens per sample (C_full)
 *   layer_gate_out  [B, L], group_gate_out [B, L, G] uint8, device: the
 *                   gates used (prefix layers on)
 *   gate_logits_out [B, L - P, G] float32, device, or NULL
 *   sample_flags    [B] uint32, device, or NULL: SVL_FLAG_GROUPS_DROPPED /
 *                   SVL_FLAG_OVER_BUDGET or-ed in by the projection
 * Other arguments as svl_gated_prefill (t_cap counts the budget-token rows).
 * Errors: as svl_gated_prefill; SVL_ERR_UNSUPPORTED without the controller
 * weights. */
svl_status svl_controlled_prefill(svl_model* model, int32_t B, int32_t t_cap, void* X, const int32_t* cu_seqlens,
                                  const int32_t* pos, const float* budget, const float* kappa, const int32_t* k,
                                  const int32_t* vis_off, const int32_t* text_len, int32_t project,
                                  int32_t logits_mode, float* logits, uint8_t* layer_gate_out,
                                  uint8_t* group_gate_out, float* gate_logits_out, uint32_t* sample_flags,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Gated decode with a KV cache (the paper leaves decode open, Sec. 5). Each
 * sample keeps its prefill gates: a gated-off head group has no cached keys
 * or values and no compute, a skipped layer is bypassed.
 *
 * The cache is caller-owned device memory, 16-byte aligned:
 *   K then V, each [L][B][max_len][A_kv * d_head] bf16; position p of
 *   sample b at row p. max_len <= the model's max_seq (RoPE table).
 * svl_kv_cache_size: its bytes (0 on bad arguments). */
size_t svl_kv_cache_size(const svl_model* model, int32_t B, int32_t max_len);

/* e4m3 quantisation of bf16 rows, as the SVL_GEMM_E4M3 path applies it to
 * weight output channels and activation rows. For each of the `rows` rows
 * of `cols` values (device bf16, `ld_src` elements apart), with
 * x = src[r, c] * gain[c] (float32, exact; gain is a device bf16 [cols]
 * vector, or NULL for x = src[r, c]): amax = max |x|, inv = 448 / amax and
 * scale[r] = amax / 448 in float32 with correct rounding (both 0 when amax
 * is 0), and dst[r * ld_dst + c] = e4m3(x * inv) rounded to nearest even and
 * saturated to +-448 (OCP e4m3: 4 exponent bits with bias 7, 3 mantissa
 * bits, no infinities). The prefill quantises the QKV and gate/up inputs
 * with their RMSNorm gain this way (the norm's 1/rms is a factor of the row,
 * applied after the product). dst is device uint8 codes, scale device
 * float32 [rows]; the caller owns both. Requires cols and ld_src multiples
 * of 8, ld_dst >= cols and a multiple of 8, src (and gain) 16-byte and dst
 * 8-byte aligned (else SVL_ERR_INVALID_ARG). Asynchronous on `stream`. */
svl_status svl_quantize_rows_e4m3(const void* src, const void* gain, int64_t rows, int32_t cols, int64_t ld_src,
                                  void* dst, int64_t ld_dst, float* scale, void* stream);

/* The e4m3 GEMM of the gated projections on its own, with an fp32 output:
 * C[m, n] = a_scale[m] * b_scale[n] * sum_k A[m, k] B[n, k], A [M, K] and
 * B [N, K] device uint8 e4m3 codes (row-major, K contiguous, 16-byte
 * aligned), scales float32, C float32 [M, N] row-major; all caller-owned.
 * Requires K a multiple of 128 and N a multiple of 32 (else
 * SVL_ERR_INVALID_ARG). The model supplies the device status word and the
 * SM count only. Asynchronous on `stream`. */
svl_status svl_gemm_e4m3(svl_model* model, const void* A, const float* a_scale, const void* B, const float* b_scale,
                         int32_t M, int32_t N, int32_t K, float* C, void* stream);

/* svl_gated_prefill that also stores every layer's keys and values of the
 * prompt into the cache and writes cache_len[B] (device int32) = the prompt
 * length S_b of each sample. Errors: as svl_gated_prefill; prompt rows past
 * max_len are not stored. */
svl_status svl_gated_prefill_kv(svl_model* model, int32_t B, int32_t t_cap, void* X, const int32_t* cu_seqlens,
                                const int32_t* pos, const uint8_t* layer_gate, const uint8_t* group_gate,
                                int32_t logits_mode, float* logits, void* kv_cache, int32_t max_len,
                                int32_t* cache_len, void* workspace, size_t workspace_bytes, void* stream);

/* One decode step: token tokens[b] (device int32 [B]) is fed to sample b at
 * position cache_len[b]; its keys and values are appended to the cache, it
 * attends to positions 0..cache_len[b] under the sample's gates
 * (layer_gate [B, L], group_gate [B, L, G] as for the prefill), logits[B, V]
 * (float32) are those of the new position, next_token[B] (device int32, or
 * NULL) the largest logit (equal logits: lower id), and cache_len[b] is
 * advanced by one. Workspace: svl_decode_workspace_size(model, B) bytes.
 * A fed id outside [0, V) or a full cache sets SVL_DEV_BAD_INDEX (the id is
 * read as 0). A sample whose cache is full (cache_len[b] >= max_len) takes
 * no step: nothing is appended, its attention output is zero, cache_len[b]
 * stays at max_len and next_token[b] is -1. Check the status word after the
 * steps of a batch. */
size_t svl_decode_workspace_size(const svl_model* model, int32_t B);
svl_status svl_decode_step(svl_model* model, int32_t B, const int32_t* tokens, void* kv_cache, int32_t max_len,
                           int32_t* cache_len, const uint8_t* layer_gate, const uint8_t* group_gate, float* logits,
                           int32_t* next_token, void* workspace, size_t workspace_bytes, void* stream);

/* svl_score_select without a workspace argument. The paper has no
 *  counterpart: this exists for callers that cannot allocate device memory
 *  for a workspace -- code running during CUDA stream capture (where
 *  cudaMalloc is not permitted), plugins whose host framework keeps all
 *  device memory for its own allocator, real-time paths that must not wait
 *  in an allocator. It allocates nothing; its scratch (budget embeddings and
 *  per-sample kept lists) lives in one fixed 512 KiB device array inside the
 *  library, present on every GPU that loads the library until the process
 *  exits. Limits: B <= 256, n_vis_total <= 65536, h_ctrl <= 256; larger
 *  calls return SVL_ERR_SHAPE and launch nothing. Outputs and their meaning
 *  are those of svl_score_select. The first call on a device looks up the
 *  array's device address (cudaGetSymbolAddress, once per device, with that
 *  device current and equal to the model's), so make that first call before
 *  any stream capture. All calls share the one array and it keeps the last
 *  call's contents; every scratch value a call reads it writes first, so
 *  nothing needs clearing, but calls that overlap on the GPU (e.g. on two
 *  streams at once) race on it and must be serialised by the caller. */
svl_status svl_score_select_noalloc(svl_model* model, int32_t B, int32_t n_vis_total,
                                    const void* vis_feats, const int32_t* vis_off, const int32_t* text_len,
                                    const float* budget, const int32_t* keep_count,
                                    const uint8_t* layer_gate, const uint8_t* group_gate,
                                    float* scores, int32_t* k, int32_t* kept_idx, int32_t* kept_off,
                                    uint32_t* sample_flags, void* stream);

/* (2) Pack (Sec. 3 S = S_text + S_vis; Sec. 3.1 contiguous RoPE).
 *  Sample b's sequence is its kept visual tokens in ascending index order,
 *  projected by the LLaVA MLP W_p2 GELU(W_p1 x) (identity when proj_hidden
 *  is 0), followed by the embeddings of its text ids; positions 0..S_b-1.
 *   text_ids [n_text_total] int32, text_off [B+1] int32
 *  Outputs: X [T_cap, D] bf16 with T_cap = n_vis_total + n_text_total (rows
 *  beyond T = sum S_b untouched), cu_seqlens [B+1] int32, pos [T_cap] int32. */
svl_status svl_pack(svl_model* model, int32_t B, int32_t n_vis_total, int32_t n_text_total,
                    const void* vis_feats, const int32_t* vis_off, const int32_t* kept_idx,
                    const int32_t* kept_off, const int32_t* text_ids, const int32_t* text_off,
                    void* X, int32_t* cu_seqlens, int32_t* pos,
                    void* workspace, size_t workspace_bytes, void* stream);

#define SVL_LOGITS_LAST 0 /* logits of each sample's last row: [B, V] */
#define SVL_LOGITS_ALL 1  /* logits of every row: [T_cap, V] */

/* (3) Gated decoder forward (Sec. 3.2; Eq. 3; Eq. 8).
 *  For each layer l and sample b with e_{b,l,j} = (l < P) or
 *  (layer_gate[b,l] and group_gate[b,l,j]): RMSNorm; Q,K,V for the heads of
 *  active groups only, with RoPE; causal attention per active head; output
 *  projection over the active heads' rows of W_O added to X; RMSNorm; SwiGLU
 *  over the active groups' FFN channels only; down projection added to X.
 *  A sample with no active group in a layer is left untouched (residual
 *  bypass). Then the final RMSNorm and the LM head. X is updated in place
 *  (on return it holds the final hidden state before the final norm).
 *   X [T_cap, D] bf16 in/out; cu_seqlens [B+1]; pos [T_cap] (from svl_pack)
 *   logits float32 [B, V] (LAST) or [T_cap, V] (ALL)
 *   t_cap: rows of X (n_vis_total + n_text_total of the pack call)
 *  B <= 4096 samples per call (else SVL_ERR_UNSUPPORTED). */
svl_status svl_gated_prefill(svl_model* model, int32_t B, int32_t t_cap, void* X,
                             const int32_t* cu_seqlens, const int32_t* pos,
                             const uint8_t* layer_gate, const uint8_t* group_gate,
                             int32_t logits_mode, float* logits,
                             void* workspace, size_t workspace_bytes, void* stream);

/* One stage of decoder layer `layer` of (3) on caller buffers: the layer
 * piecewise, with exactly the kernels and launch configuration the prefill
 * uses (the stage inside svl_gated_prefill is the same code path). Serves
 * per-stage checks of a layer and callers that interleave their own work
 * between the stages. Gates, cu_seqlens, pos, t_cap and the workspace are as
 * for svl_gated_prefill (a workspace sized for the prefill suffices); the
 * RMSNorm sums of squares that the prefill carries from the previous stage
 * are recomputed from X. d_h = D / A, t_pad = t_cap rounded up to 8.
 *  SVL_LAYER_QKV:    X -> q [t_cap, A*d_h], k [t_cap, A_kv*d_h] (RoPE at pos)
 *                    and vt [A_kv*d_h, t_pad] (V transposed), for the heads of
 *                    active groups (other columns untouched)
 *  SVL_LAYER_ATTN:   q, k, vt -> ao [t_cap, A*d_h]: causal attention of the
 *                    active heads (key columns of vt past the packed rows
 *                    must hold finite values)
 *  SVL_LAYER_OPROJ:  X += ao W_O^T over the active heads' rows of W_O
 *  SVL_LAYER_GATEUP: X -> h [t_cap, D_int] = SiLU(xn W_g^T) * (xn W_u^T),
 *                    xn = RMSNorm(X) * gain, active groups' channels only
 *  SVL_LAYER_DOWN:   X += h W_down^T over the active channels
 * Buffers a stage does not use may be NULL. All bf16, device, caller-owned,
 * 16-byte aligned. Errors: as svl_gated_prefill; a bad stage or layer, or a
 * missing buffer the stage needs: SVL_ERR_INVALID_ARG. */
#define SVL_LAYER_QKV 0
#define SVL_LAYER_ATTN 1
#define SVL_LAYER_OPROJ 2
#define SVL_LAYER_GATEUP 3
#define SVL_LAYER_DOWN 4
svl_status svl_layer_stage(svl_model* model, int32_t stage, int32_t layer, int32_t B, int32_t t_cap, void* X,
                           const int32_t* cu_seqlens, const int32_t* pos, const uint8_t* layer_gate,
                           const uint8_t* group_gate, void* q, void* k, void* vt, void* ao, void* h,
                           void* workspace, size_t workspace_bytes, void* stream);

/* Eq. 8 for one sample, host only, no GPU: writes G * C(S) (exact integer
 * arithmetic, 8 D^2 generalised to 4 D^2 + 4 D D_kv) for S = s_text + s_vis
 * with the gates given (layer_gate [L], group_gate [L, G]; NULL = all on),
 * and the FLOPs the gated path executes (causal attention, last-row logits). */
svl_status svl_flops(const svl_model_desc* desc, int32_t s_text, int32_t s_vis, int32_t n_vis,
                     const uint8_t* layer_gate, const uint8_t* group_gate,
                     double* eq8_flops, double* exec_flops);

/* End to end from HOST buffers: copies the inputs of one batch to the device
 *  (asynchronously on `stream`; pinned host memory makes the copies
 *  overlap), runs svl_score_select, svl_pack and svl_gated_prefill (LAST
 *  logits) and copies the logits [B, V] float32 and k [B] int32 back to the
 *  host buffers. The caller synchronises `stream` before reading them.
 *  Host inputs are laid out as the device arguments of (1) and (2):
 *  h_vis [n_vis_total, C_v] bf16, h_vis_off [B+1], h_text_ids
 *  [n_text_total], h_text_off [B+1], h_budget [B], h_keep_count [B] or NULL,
 *  h_layer_gate [B, L], h_group_gate [B, L, G]. `workspace` must hold
 *  svl_host_workspace_size() bytes for these sizes. */
svl_status svl_prefill_from_host(svl_model* model, int32_t B, int32_t n_vis_total, int32_t n_text_total,
                                 const void* h_vis, const int32_t* h_vis_off, const int32_t* h_text_ids,
                                 const int32_t* h_text_off, const float* h_budget, const int32_t* h_keep_count,
                                 const uint8_t* h_layer_gate, const uint8_t* h_group_gate,
                                 float* h_logits, int32_t* h_k,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* Workspace bytes of svl_prefill_from_host for these sizes. */
size_t svl_host_workspace_size(const svl_model* model, int32_t B, int64_t n_vis_total, int64_t n_text_total);

/* Kernel timing. While profiling is on, the library records a CUDA event
 * pair on the launch stream around every kernel it launches whose tag bit is
 * set in `tag_mask`, tagged by the step of the path (events between kernels
 * keep a kernel from starting before its predecessor finishes, so record
 * only what is needed while timing end to end). svl_profile_stop() waits for the last event, sums the
 * elapsed times per tag into `out` (at most `cap` entries, *n_out set) and
 * turns profiling off. */
typedef struct svl_kernel_time {
  int32_t tag;       /* SVL_TAG_* */
  int32_t launches;
  double total_ms;
} svl_kernel_time;

#define SVL_TAG_BUDGET_EMBED 0
#define SVL_TAG_SCORE 1
#define SVL_TAG_SELECT 2
#define SVL_TAG_PACK 3
#define SVL_TAG_PROJECTOR 4
#define SVL_TAG_SCHEDULE 5
#define SVL_TAG_RMSNORM 6
#define SVL_TAG_QKV 7
#define SVL_TAG_ATTENTION 8
#define SVL_TAG_OPROJ 9
#define SVL_TAG_GATEUP 10
#define SVL_TAG_DOWN 11
#define SVL_TAG_LMHEAD 12
#define SVL_TAG_COPY 13
#define SVL_TAG_QUANT 14 /* e4m3 quantisation of the gated GEMMs' activation rows */
#define SVL_TAG_COUNT 15

svl_status svl_profile_start(svl_model* model, uint32_t tag_mask); /* bit t: record SVL_TAG t */
svl_status svl_profile_stop(svl_model* model, svl_kernel_time* out, int32_t cap, int32_t* n_out);
/* The individual launches of the last profiling window (after
 * svl_profile_stop), in launch order: tag and elapsed milliseconds of each.
 * Writes at most `cap` entries and sets *n_out to the number written. */
svl_status svl_profile_launches(svl_model* model, int32_t* tags, float* ms, int32_t cap, int32_t* n_out);
const char* svl_tag_name(int32_t tag);

/* Self-test of the device-side time-out path (the paper has no
 * counterpart): launches one CTA that waits on a shared-memory barrier that
 * nothing ever arrives on, giving up after `wait_cycles` SM clock cycles the
 * way every wait in the library does, so SVL_DEV_TIMEOUT is set in the
 * status word and the kernel returns normally. `wait_cycles` is clamped to
 * [1000, 1e9]. Asynchronous on `stream`. */
svl_status svl_selftest_wait_timeout(svl_model* model, uint64_t wait_cycles, void* stream);

/* Reads (and clears) the device status word; synchronises `stream`. */
svl_status svl_get_device_status(svl_model* model, void* stream, uint32_t* code);

const char* svl_status_string(svl_status s);

/* Number of kernels launched by this library since the process started
 * (host-side counter, used to report launches per step). */
uint64_t svl_launch_count(void);

/* The launch rule of the residual GEMMs' K-split tail, host only (no GPU):
 * the number of K shares (1 = no split) the last wave of a residual GEMM
 * list of `tiles` tiles (list capacity `cap`) is cut into, on a persistent
 * grid of num_sms CTAs of which blocks_per_sm fit on one SM, with `units`
 * partial tiles of workspace. The shares wait for each other inside one
 * launch, so the tail is split only when the whole grid is resident at once
 * (blocks_per_sm >= 1); svl_model_create queries the occupancy of the
 * residual GEMM and the prefill disables the split when it is 0. Beyond
 * that: a last wave of r = tiles % num_sms tiles is split only when
 * 0 < r <= num_sms / 2, into min(num_sms / r, 8, units / r,
 * 1 + (cap - tiles) / r) shares, if that is at least 2. The paper has no
 * counterpart; this is the library's load balancing of partial waves. */
int32_t svl_ksplit_plan(int32_t tiles, int32_t cap, int32_t num_sms, int32_t blocks_per_sm, int32_t units);

#ifdef __cplusplus
}
#endif
#endif /* SVL_H */
