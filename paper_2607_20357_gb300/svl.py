"""Python binding of libsvl.so (ctypes): the C ABI of ``include/svl.h``.

Every function here only marshals arguments -- torch tensors become device
pointers, the stream is torch's current CUDA stream -- and calls the C entry
point of the same name. All computation runs in the library's CUDA kernels.
There is no fallback: if the library is missing or fails to load, the call
raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsvl.so")
_lib = None

SVL_LOGITS_LAST = 0
SVL_LOGITS_ALL = 1
SVL_FLAG_OVER_BUDGET = 1
SVL_FLAG_GROUPS_DROPPED = 2
SVL_DEV_NONFINITE, SVL_DEV_TIMEOUT, SVL_DEV_BAD_INDEX = 1, 2, 4
SVL_GEMM_BF16, SVL_GEMM_E4M3 = 0, 1
SVL_LAYER_QKV, SVL_LAYER_ATTN, SVL_LAYER_OPROJ, SVL_LAYER_GATEUP, SVL_LAYER_DOWN = 0, 1, 2, 3, 4

SYMBOLS = ["svl_model_create", "svl_model_destroy", "svl_workspace_size", "svl_score_select", "svl_pack",
           "svl_gated_prefill", "svl_flops", "svl_get_device_status", "svl_status_string", "svl_launch_count",
           "svl_prefill_from_host", "svl_host_workspace_size", "svl_profile_start", "svl_profile_stop",
           "svl_tag_name", "svl_score_select_noalloc", "svl_profile_launches", "svl_selftest_wait_timeout",
           "svl_workspace_size_for", "svl_score_select_paper", "svl_pack_controlled", "svl_controlled_prefill",
           "svl_kv_cache_size", "svl_gated_prefill_kv", "svl_decode_workspace_size", "svl_decode_step",
           "svl_quantize_rows_e4m3", "svl_gemm_e4m3", "svl_layer_stage", "svl_ksplit_plan"]

TAGS = ["budget_embed", "score", "select", "pack", "projector", "schedule", "rmsnorm", "qkv_gemm", "attention",
        "o_gemm", "gateup_gemm", "down_gemm", "lm_head", "host_copy", "quant"]


class KernelTime(ctypes.Structure):
    _fields_ = [("tag", ctypes.c_int32), ("launches", ctypes.c_int32), ("total_ms", ctypes.c_double)]


class ModelDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("n_layers", "d_model", "n_heads", "n_kv_heads", "d_ffn", "vocab",
                                              "n_groups", "n_prefix", "c_vis", "h_ctrl", "proj_hidden")] + \
               [("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float), ("max_seq", ctypes.c_int32),
                ("gemm_format", ctypes.c_int32)]


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("wq", "wk", "wv", "wo", "wg", "wu", "wd", "attn_norm", "ffn_norm")]


class Weights(ctypes.Structure):
    _fields_ = [("ctrl_w1", ctypes.c_void_p), ("ctrl_w2", ctypes.c_void_p), ("ctrl_c2", ctypes.c_float),
                ("bud_w1", ctypes.c_void_p), ("bud_w2", ctypes.c_void_p), ("proj_w1", ctypes.c_void_p),
                ("proj_w2", ctypes.c_void_p), ("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p), ("layers", ctypes.POINTER(LayerWeights)),
                ("llm_bud_w1", ctypes.c_void_p), ("llm_bud_w2", ctypes.c_void_p), ("kap_w1", ctypes.c_void_p),
                ("kap_w2", ctypes.c_void_p), ("gate_w", ctypes.c_void_p), ("gate_c", ctypes.c_void_p)]


def lib():
    """Loads libsvl.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libsvl.so not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        L.svl_model_create.argtypes = [ctypes.POINTER(ModelDesc), ctypes.POINTER(Weights), ctypes.POINTER(vp)]
        L.svl_model_create.restype = ctypes.c_int
        L.svl_model_destroy.argtypes = [vp]
        L.svl_model_destroy.restype = None
        L.svl_workspace_size.argtypes = [vp, i32, i64, i64]
        L.svl_workspace_size.restype = sz
        L.svl_score_select.argtypes = [vp, i32, i32] + [vp] * 13 + [sz, vp]
        L.svl_score_select.restype = ctypes.c_int
        L.svl_pack.argtypes = [vp, i32, i32, i32] + [vp] * 10 + [sz, vp]
        L.svl_pack.restype = ctypes.c_int
        L.svl_gated_prefill.argtypes = [vp, i32, i32, vp, vp, vp, vp, vp, i32, vp, vp, sz, vp]
        L.svl_gated_prefill.restype = ctypes.c_int
        L.svl_flops.argtypes = [ctypes.POINTER(ModelDesc), i32, i32, i32, vp, vp,
                                ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]
        L.svl_flops.restype = ctypes.c_int
        L.svl_get_device_status.argtypes = [vp, vp, ctypes.POINTER(ctypes.c_uint32)]
        L.svl_get_device_status.restype = ctypes.c_int
        L.svl_status_string.argtypes = [ctypes.c_int]
        L.svl_status_string.restype = ctypes.c_char_p
        L.svl_launch_count.argtypes = []
        L.svl_launch_count.restype = ctypes.c_uint64
        L.svl_prefill_from_host.argtypes = [vp, i32, i32, i32] + [vp] * 11 + [sz, vp]
        L.svl_prefill_from_host.restype = ctypes.c_int
        L.svl_host_workspace_size.argtypes = [vp, i32, i64, i64]
        L.svl_host_workspace_size.restype = sz
        L.svl_profile_start.argtypes = [vp, ctypes.c_uint32]
        L.svl_profile_start.restype = ctypes.c_int
        L.svl_profile_stop.argtypes = [vp, ctypes.POINTER(KernelTime), i32, ctypes.POINTER(i32)]
        L.svl_profile_stop.restype = ctypes.c_int
        L.svl_tag_name.argtypes = [i32]
        L.svl_tag_name.restype = ctypes.c_char_p
        L.svl_score_select_paper.argtypes = [vp, i32, i32] + [vp] * 15 + [sz, vp]
        L.svl_score_select_paper.restype = ctypes.c_int
        L.svl_pack_controlled.argtypes = [vp, i32, i32, i32] + [vp] * 11 + [sz, vp]
        L.svl_pack_controlled.restype = ctypes.c_int
        L.svl_controlled_prefill.argtypes = [vp, i32, i32] + [vp] * 8 + [i32, i32] + [vp] * 6 + [sz, vp]
        L.svl_controlled_prefill.restype = ctypes.c_int
        L.svl_kv_cache_size.argtypes = [vp, i32, i32]
        L.svl_kv_cache_size.restype = sz
        L.svl_gated_prefill_kv.argtypes = [vp, i32, i32, vp, vp, vp, vp, vp, i32, vp, vp, i32, vp, vp, sz, vp]
        L.svl_gated_prefill_kv.restype = ctypes.c_int
        L.svl_decode_workspace_size.argtypes = [vp, i32]
        L.svl_decode_workspace_size.restype = sz
        L.svl_decode_step.argtypes = [vp, i32, vp, vp, i32] + [vp] * 6 + [sz, vp]
        L.svl_decode_step.restype = ctypes.c_int
        L.svl_score_select_noalloc.argtypes = [vp, i32, i32] + [vp] * 13
        L.svl_score_select_noalloc.restype = ctypes.c_int
        L.svl_profile_launches.argtypes = [vp, ctypes.POINTER(i32), ctypes.POINTER(ctypes.c_float), i32,
                                           ctypes.POINTER(i32)]
        L.svl_profile_launches.restype = ctypes.c_int
        L.svl_selftest_wait_timeout.argtypes = [vp, ctypes.c_uint64, vp]
        L.svl_selftest_wait_timeout.restype = ctypes.c_int
        L.svl_workspace_size_for.argtypes = [vp, ctypes.c_uint32, i32, i64, i64]
        L.svl_workspace_size_for.restype = sz
        L.svl_quantize_rows_e4m3.argtypes = [vp, vp, i64, i32, i64, vp, i64, vp, vp]
        L.svl_quantize_rows_e4m3.restype = ctypes.c_int
        L.svl_gemm_e4m3.argtypes = [vp] * 5 + [i32, i32, i32, vp, vp]
        L.svl_gemm_e4m3.restype = ctypes.c_int
        L.svl_layer_stage.argtypes = [vp, i32, i32, i32, i32] + [vp] * 10 + [vp, sz, vp]
        L.svl_layer_stage.restype = ctypes.c_int
        L.svl_ksplit_plan.argtypes = [i32] * 5
        L.svl_ksplit_plan.restype = i32
        _lib = L
    return _lib


class SvlError(RuntimeError):
    def __init__(self, fn, code):
        super().__init__(f"{fn}: {lib().svl_status_string(code).decode()} (status {code})")
        self.code = code


def _check(fn, code):
    if code != 0:
        raise SvlError(fn, code)


def _p(x):
    """Device (or host) pointer of a tensor / int / None."""
    if x is None:
        return None
    if isinstance(x, torch.Tensor):
        return ctypes.c_void_p(x.data_ptr())
    return ctypes.c_void_p(int(x))


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def svl_model_create(desc: ModelDesc, weights: Weights):
    h = ctypes.c_void_p()
    _check("svl_model_create", lib().svl_model_create(ctypes.byref(desc), ctypes.byref(weights), ctypes.byref(h)))
    return h


def svl_model_destroy(model):
    lib().svl_model_destroy(model)


def svl_workspace_size(model, max_batch, max_vis_total, max_text_total) -> int:
    return int(lib().svl_workspace_size(model, int(max_batch), int(max_vis_total), int(max_text_total)))


STAGE_BITS = {"select": 1, "pack": 2, "prefill": 4}


def svl_workspace_size_for(model, stages, max_batch, max_vis_total, max_text_total) -> int:
    mask = sum(STAGE_BITS[s] for s in stages)
    return int(lib().svl_workspace_size_for(model, ctypes.c_uint32(mask), int(max_batch), int(max_vis_total),
                                            int(max_text_total)))


def svl_score_select(model, B, n_vis_total, vis_feats, vis_off, text_len, budget, keep_count, layer_gate,
                     group_gate, scores, k, kept_idx, kept_off, sample_flags, workspace, workspace_bytes,
                     stream=None):
    _check("svl_score_select", lib().svl_score_select(
        model, int(B), int(n_vis_total), _p(vis_feats), _p(vis_off), _p(text_len), _p(budget), _p(keep_count),
        _p(layer_gate), _p(group_gate), _p(scores), _p(k), _p(kept_idx), _p(kept_off), _p(sample_flags),
        _p(workspace), int(workspace_bytes), _stream(stream)))


def svl_score_select_paper(model, B, n_vis_total, vis_feats, vis_off, text_len, budget, keep_count, gate_logits,
                           scores, k, kept_idx, kept_off, sample_flags, layer_gate_out, group_gate_out, kappa_out,
                           workspace, workspace_bytes, stream=None):
    """The paper's own inference rule (sigma(z) > 0.5 tokens, gates from the
    compute controller's logits or decided later, budget projection): see svl.h."""
    _check("svl_score_select_paper", lib().svl_score_select_paper(
        model, int(B), int(n_vis_total), _p(vis_feats), _p(vis_off), _p(text_len), _p(budget), _p(keep_count),
        _p(gate_logits), _p(scores), _p(k), _p(kept_idx), _p(kept_off), _p(sample_flags), _p(layer_gate_out),
        _p(group_gate_out), _p(kappa_out), _p(workspace), int(workspace_bytes), _stream(stream)))


def svl_kv_cache_size(model, B, max_len) -> int:
    return int(lib().svl_kv_cache_size(model, int(B), int(max_len)))


def svl_gated_prefill_kv(model, B, t_cap, X, cu_seqlens, pos, layer_gate, group_gate, logits_mode, logits,
                         kv_cache, max_len, cache_len, workspace, workspace_bytes, stream=None):
    _check("svl_gated_prefill_kv", lib().svl_gated_prefill_kv(
        model, int(B), int(t_cap), _p(X), _p(cu_seqlens), _p(pos), _p(layer_gate), _p(group_gate),
        int(logits_mode), _p(logits), _p(kv_cache), int(max_len), _p(cache_len), _p(workspace),
        int(workspace_bytes), _stream(stream)))


def svl_quantize_rows_e4m3(src, rows, cols, ld_src, dst, ld_dst, scale, stream=None, gain=None):
    _check("svl_quantize_rows_e4m3", lib().svl_quantize_rows_e4m3(
        _p(src), _p(gain), int(rows), int(cols), int(ld_src), _p(dst), int(ld_dst), _p(scale), _stream(stream)))


def svl_gemm_e4m3(model, A, a_scale, B, b_scale, M, N, K, C, stream=None):
    _check("svl_gemm_e4m3", lib().svl_gemm_e4m3(model, _p(A), _p(a_scale), _p(B), _p(b_scale), int(M), int(N),
                                                int(K), _p(C), _stream(stream)))


def svl_layer_stage(model, stage, layer, B, t_cap, X, cu_seqlens, pos, layer_gate, group_gate, q=None, k=None,
                    vt=None, ao=None, h=None, workspace=None, workspace_bytes=0, stream=None):
    """One stage of one decoder layer on caller buffers (see svl.h)."""
    _check("svl_layer_stage", lib().svl_layer_stage(
        model, int(stage), int(layer), int(B), int(t_cap), _p(X), _p(cu_seqlens), _p(pos), _p(layer_gate),
        _p(group_gate), _p(q), _p(k), _p(vt), _p(ao), _p(h), _p(workspace), int(workspace_bytes),
        _stream(stream)))


def svl_ksplit_plan(tiles, cap, num_sms, blocks_per_sm, units) -> int:
    """K shares of a residual GEMM's last wave (1 = no split); host only."""
    return int(lib().svl_ksplit_plan(int(tiles), int(cap), int(num_sms), int(blocks_per_sm), int(units)))


def svl_decode_workspace_size(model, B) -> int:
    return int(lib().svl_decode_workspace_size(model, int(B)))


def svl_decode_step(model, B, tokens, kv_cache, max_len, cache_len, layer_gate, group_gate, logits, next_token,
                    workspace, workspace_bytes, stream=None):
    _check("svl_decode_step", lib().svl_decode_step(
        model, int(B), _p(tokens), _p(kv_cache), int(max_len), _p(cache_len), _p(layer_gate), _p(group_gate),
        _p(logits), _p(next_token), _p(workspace), int(workspace_bytes), _stream(stream)))


def svl_pack_controlled(model, B, n_vis_total, n_text_total, vis_feats, vis_off, kept_idx, kept_off, text_ids,
                        text_off, budget, X, cu_seqlens, pos, workspace, workspace_bytes, stream=None):
    _check("svl_pack_controlled", lib().svl_pack_controlled(
        model, int(B), int(n_vis_total), int(n_text_total), _p(vis_feats), _p(vis_off), _p(kept_idx),
        _p(kept_off), _p(text_ids), _p(text_off), _p(budget), _p(X), _p(cu_seqlens), _p(pos), _p(workspace),
        int(workspace_bytes), _stream(stream)))


def svl_controlled_prefill(model, B, t_cap, X, cu_seqlens, pos, budget, kappa, k, vis_off, text_len, project,
                           logits_mode, logits, layer_gate_out, group_gate_out, gate_logits_out, sample_flags,
                           workspace, workspace_bytes, stream=None):
    _check("svl_controlled_prefill", lib().svl_controlled_prefill(
        model, int(B), int(t_cap), _p(X), _p(cu_seqlens), _p(pos), _p(budget), _p(kappa), _p(k), _p(vis_off),
        _p(text_len), int(project), int(logits_mode), _p(logits), _p(layer_gate_out), _p(group_gate_out),
        _p(gate_logits_out), _p(sample_flags), _p(workspace), int(workspace_bytes), _stream(stream)))


def svl_score_select_noalloc(model, B, n_vis_total, vis_feats, vis_off, text_len, budget, keep_count, layer_gate,
                             group_gate, scores, k, kept_idx, kept_off, sample_flags, stream=None):
    """svl_score_select for callers that cannot allocate a workspace: the
    library's fixed device scratch array is used instead (see svl.h)."""
    _check("svl_score_select_noalloc", lib().svl_score_select_noalloc(
        model, int(B), int(n_vis_total), _p(vis_feats), _p(vis_off), _p(text_len), _p(budget), _p(keep_count),
        _p(layer_gate), _p(group_gate), _p(scores), _p(k), _p(kept_idx), _p(kept_off), _p(sample_flags),
        _stream(stream)))


def svl_pack(model, B, n_vis_total, n_text_total, vis_feats, vis_off, kept_idx, kept_off, text_ids, text_off,
             X, cu_seqlens, pos, workspace, workspace_bytes, stream=None):
    _check("svl_pack", lib().svl_pack(
        model, int(B), int(n_vis_total), int(n_text_total), _p(vis_feats), _p(vis_off), _p(kept_idx),
        _p(kept_off), _p(text_ids), _p(text_off), _p(X), _p(cu_seqlens), _p(pos), _p(workspace),
        int(workspace_bytes), _stream(stream)))


def svl_gated_prefill(model, B, t_cap, X, cu_seqlens, pos, layer_gate, group_gate, logits_mode, logits,
                      workspace, workspace_bytes, stream=None):
    _check("svl_gated_prefill", lib().svl_gated_prefill(
        model, int(B), int(t_cap), _p(X), _p(cu_seqlens), _p(pos), _p(layer_gate), _p(group_gate),
        int(logits_mode), _p(logits), _p(workspace), int(workspace_bytes), _stream(stream)))


def svl_flops(desc: ModelDesc, s_text, s_vis, n_vis, layer_gate=None, group_gate=None):
    """Host-side Eq. 8 (eq8) and executed FLOPs for one sample; gates are
    CPU uint8 tensors [L] and [L, G] or None (all on)."""
    eq8, ex = ctypes.c_double(), ctypes.c_double()
    lg = None if layer_gate is None else ctypes.c_void_p(layer_gate.contiguous().data_ptr())
    gg = None if group_gate is None else ctypes.c_void_p(group_gate.contiguous().data_ptr())
    _check("svl_flops", lib().svl_flops(ctypes.byref(desc), int(s_text), int(s_vis), int(n_vis), lg, gg,
                                        ctypes.byref(eq8), ctypes.byref(ex)))
    return eq8.value, ex.value


def svl_selftest_wait_timeout(model, wait_cycles=100000, stream=None):
    _check("svl_selftest_wait_timeout", lib().svl_selftest_wait_timeout(model, ctypes.c_uint64(int(wait_cycles)),
                                                                        _stream(stream)))


def svl_get_device_status(model, stream=None) -> int:
    code = ctypes.c_uint32()
    _check("svl_get_device_status", lib().svl_get_device_status(model, _stream(stream), ctypes.byref(code)))
    return int(code.value)


def svl_launch_count() -> int:
    return int(lib().svl_launch_count())


def svl_prefill_from_host(model, B, n_vis_total, n_text_total, h_vis, h_vis_off, h_text_ids, h_text_off, h_budget,
                          h_keep_count, h_layer_gate, h_group_gate, h_logits, h_k, workspace, workspace_bytes,
                          stream=None):
    """Host tensors (pinned CPU) in, host logits/k out; async on the stream."""
    _check("svl_prefill_from_host", lib().svl_prefill_from_host(
        model, int(B), int(n_vis_total), int(n_text_total), _p(h_vis), _p(h_vis_off), _p(h_text_ids),
        _p(h_text_off), _p(h_budget), _p(h_keep_count), _p(h_layer_gate), _p(h_group_gate), _p(h_logits),
        _p(h_k), _p(workspace), int(workspace_bytes), _stream(stream)))


def svl_host_workspace_size(model, B, n_vis_total, n_text_total) -> int:
    return int(lib().svl_host_workspace_size(model, int(B), int(n_vis_total), int(n_text_total)))


def svl_profile_start(model, tags=None):
    """Records events around the kernels whose tag names are in `tags`
    (default: every kernel)."""
    mask = 0xFFFFFFFF if tags is None else sum(1 << TAGS.index(t) for t in tags)
    _check("svl_profile_start", lib().svl_profile_start(model, ctypes.c_uint32(mask)))


def svl_profile_launches(model, cap=1 << 16):
    """[(tag name, ms)] of every launch of the last profiling window."""
    tags = (ctypes.c_int32 * cap)()
    ms = (ctypes.c_float * cap)()
    n = ctypes.c_int32()
    _check("svl_profile_launches", lib().svl_profile_launches(model, tags, ms, cap, ctypes.byref(n)))
    return [(TAGS[tags[i]] if 0 <= tags[i] < len(TAGS) else str(tags[i]), float(ms[i])) for i in range(n.value)]


def svl_profile_stop(model) -> dict:
    """{tag name: (launches, total ms)} of the kernels since svl_profile_start."""
    buf = (KernelTime * 32)()
    n = ctypes.c_int32()
    _check("svl_profile_stop", lib().svl_profile_stop(model, buf, 32, ctypes.byref(n)))
    return {lib().svl_tag_name(buf[i].tag).decode(): (int(buf[i].launches), float(buf[i].total_ms))
            for i in range(n.value)}


# --------------------------------------------------------------------------- plumbing
def model_desc(dims, max_seq: int, gemm_format: int = SVL_GEMM_BF16) -> ModelDesc:
    return ModelDesc(n_layers=dims.n_layers, d_model=dims.d_model, n_heads=dims.n_heads,
                     n_kv_heads=dims.n_kv_heads, d_ffn=dims.d_ffn, vocab=dims.vocab, n_groups=dims.n_groups,
                     n_prefix=dims.n_prefix, c_vis=dims.c_vis, h_ctrl=dims.h_ctrl, proj_hidden=dims.proj_hidden,
                     rms_eps=dims.rms_eps, rope_theta=dims.rope_theta, max_seq=int(max_seq),
                     gemm_format=int(gemm_format))


class GatedPrefill:
    """Owns a model handle and the device weight tensors it points to.

    ``weights`` is a dict as produced by the input generator, tensors on the
    CUDA device (bf16, nn.Linear layout). ``run`` allocates the outputs and
    the workspace with torch and calls the three C entry points in order.
    ``gemm_format`` = SVL_GEMM_E4M3 runs the gated projections on e4m3
    operands (the model quantises its weights once, at creation).
    """

    def __init__(self, dims, weights: dict, max_seq: int = 8192, gemm_format: int = SVL_GEMM_BF16):
        self.dims = dims
        self.w = weights
        self.desc = model_desc(dims, max_seq, gemm_format)
        lw = (LayerWeights * dims.n_layers)()
        for i, l in enumerate(weights["layers"]):
            lw[i] = LayerWeights(*[l[n].data_ptr() for n in ("wq", "wk", "wv", "wo", "wg", "wu", "wd",
                                                             "attn_norm", "ffn_norm")])
        self._lw = lw
        opt = lambda n: weights[n].data_ptr() if n in weights else None
        self._wts = Weights(weights["ctrl_w1"].data_ptr(), weights["ctrl_w2"].data_ptr(), float(weights["ctrl_c2"]),
                            weights["bud_w1"].data_ptr(), weights["bud_w2"].data_ptr(), opt("proj_w1"),
                            opt("proj_w2"), weights["embed"].data_ptr(), weights["final_norm"].data_ptr(),
                            weights["lm_head"].data_ptr(), lw, opt("llm_bud_w1"), opt("llm_bud_w2"), opt("kap_w1"),
                            opt("kap_w2"), opt("gate_w"), opt("gate_c"))
        self.handle = svl_model_create(self.desc, self._wts)
        self._ws = None
        self._ws_key = None

    def close(self):
        if self.handle:
            svl_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def workspace(self, B, n_vis, n_text, device="cuda", stages=("select", "pack", "prefill")):
        need = svl_workspace_size_for(self.handle, stages, B, n_vis, n_text)
        if self._ws is None or self._ws.numel() < need:
            self._ws = torch.empty(need, dtype=torch.uint8, device=device)
        return self._ws, self._ws.numel()

    def alloc_outputs(self, batch: dict, logits_mode: int = SVL_LOGITS_LAST):
        d = self.dims
        B = batch["B"]
        nv = batch["vis"].shape[0]
        nt = int(batch["text_ids"].shape[0])
        dev = batch["vis"].device
        t_cap = nv + nt + B  # room for one budget-token row per sample (rule="controller")
        i32 = dict(dtype=torch.int32, device=dev)
        return {
            "scores": torch.empty(max(nv, 1), dtype=torch.float32, device=dev),
            "k": torch.empty(B, **i32),
            "kept_idx": torch.empty(max(nv, 1), **i32),
            "kept_off": torch.empty(B + 1, **i32),
            "flags": torch.empty(B, dtype=torch.int32, device=dev),
            "X": torch.empty(max(t_cap, 1), d.d_model, dtype=torch.bfloat16, device=dev),
            "cu_seqlens": torch.empty(B + 1, **i32),
            "pos": torch.empty(max(t_cap, 1), **i32),
            "logits": torch.empty((B if logits_mode == SVL_LOGITS_LAST else max(t_cap, 1)), d.vocab,
                                  dtype=torch.float32, device=dev),
            "text_len": (batch["text_off"][1:] - batch["text_off"][:-1]).to(torch.int32).contiguous(),
            # projected gates of the paper's rule (rule="paper") or the controller's (rule="controller")
            "layer_gate": torch.empty(B, d.n_layers, dtype=torch.uint8, device=dev),
            "group_gate": torch.empty(B, d.n_layers, d.n_groups, dtype=torch.uint8, device=dev),
            "kappa": torch.empty(B, dtype=torch.float32, device=dev),
            "gate_logits": torch.empty(B, max(d.n_layers - d.n_prefix, 1), d.n_groups, dtype=torch.float32,
                                       device=dev),
        }

    def _run_controlled(self, batch, out, logits_mode, stream, stages, ws, wsb, nv, nt):
        B = batch["B"]
        if "select" in stages:
            svl_score_select_paper(self.handle, B, nv, batch["vis"], batch["vis_off"], out["text_len"],
                                   batch["budget"], batch["keep_count"], None, out["scores"], out["k"],
                                   out["kept_idx"], out["kept_off"], out["flags"], None, None, out["kappa"], ws, wsb,
                                   stream)
        if "pack" in stages:
            svl_pack_controlled(self.handle, B, nv, nt, batch["vis"], batch["vis_off"], out["kept_idx"],
                                out["kept_off"], batch["text_ids"], batch["text_off"], batch["budget"], out["X"],
                                out["cu_seqlens"], out["pos"], ws, wsb, stream)
        if "prefill" in stages:
            svl_controlled_prefill(self.handle, B, nv + nt + B, out["X"], out["cu_seqlens"], out["pos"],
                                   batch["budget"], out["kappa"], out["k"], batch["vis_off"], out["text_len"], 1,
                                   logits_mode, out["logits"], out["layer_gate"], out["group_gate"],
                                   out["gate_logits"], out["flags"], ws, wsb, stream)
        return out

    def run(self, batch: dict, out: Optional[dict] = None, logits_mode: int = SVL_LOGITS_LAST, stream=None,
            stages=("select", "pack", "prefill"), rule: str = "budget"):
        """rule="budget": k from the budget for the given gates (the hot path);
        rule="paper": the paper's own inference rule from batch["gate_logits"]
        ([B, L, G] compute-controller logits), whose projected gates (in
        out["layer_gate"], out["group_gate"]) then drive the prefill;
        rule="controller": tokens with z > 0, the budget token appended, and
        the compute controller deciding the gates on the device after the
        prefix layers (out["kappa"], out["gate_logits"], out gates)."""
        B = batch["B"]
        nv = batch["vis"].shape[0]
        nt = int(batch["text_ids"].shape[0])
        out = out or self.alloc_outputs(batch, logits_mode)
        ws, wsb = self.workspace(B, nv, nt, batch["vis"].device, stages)
        if rule not in ("budget", "paper", "controller"):
            raise ValueError(f"unknown rule {rule!r}")
        if rule == "controller":
            return self._run_controlled(batch, out, logits_mode, stream, stages, ws, wsb, nv, nt)
        gates = (out["layer_gate"], out["group_gate"]) if rule == "paper" else (batch["layer_gate"], batch["group_gate"])
        if "select" in stages and rule == "paper":
            svl_score_select_paper(self.handle, B, nv, batch["vis"], batch["vis_off"], out["text_len"],
                                   batch["budget"], batch["keep_count"], batch["gate_logits"], out["scores"],
                                   out["k"], out["kept_idx"], out["kept_off"], out["flags"], out["layer_gate"],
                                   out["group_gate"], out["kappa"], ws, wsb, stream)
        elif "select" in stages:
            svl_score_select(self.handle, B, nv, batch["vis"], batch["vis_off"], out["text_len"], batch["budget"],
                             batch["keep_count"], batch["layer_gate"], batch["group_gate"], out["scores"], out["k"],
                             out["kept_idx"], out["kept_off"], out["flags"], ws, wsb, stream)
        if "pack" in stages:
            svl_pack(self.handle, B, nv, nt, batch["vis"], batch["vis_off"], out["kept_idx"], out["kept_off"],
                     batch["text_ids"], batch["text_off"], out["X"], out["cu_seqlens"], out["pos"], ws, wsb, stream)
        if "prefill" in stages:
            svl_gated_prefill(self.handle, B, max(nv + nt, 1), out["X"], out["cu_seqlens"], out["pos"],
                              gates[0], gates[1], logits_mode, out["logits"], ws, wsb, stream)
        return out
