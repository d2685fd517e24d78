"""ctypes binding of the C ABI in include/mmshift.h (argument marshalling only).

Every function here forwards to the entry point of the same name in
libmmshift.so; all computation happens in the library's CUDA kernels. The
library is built in-tree by ``paper_2607_22586_gb300.build`` and loading fails
loudly if it cannot be built or found.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

from . import build as _build

MMSHIFT_OK = 0
MMSHIFT_ERR_INVALID_ARG = 1
MMSHIFT_ERR_UNSUPPORTED = 2
MMSHIFT_ERR_WORKSPACE = 3
MMSHIFT_ERR_CUDA = 4
MMSHIFT_ERR_TIMEOUT = 5
MMSHIFT_ERR_DEVICE = 6

MMSHIFT_BF16 = 0
MMSHIFT_F32 = 1
MMSHIFT_SCORE_VOTE = 0
MMSHIFT_SCORE_MASS = 1
MMSHIFT_MAX_BATCH = 64

EXPORTED = [
    "mmshift_default_params", "mmshift_output_rows", "mmshift_workspace_size",
    "mmshift_build_proxies", "mmshift_proxy_mass", "mmshift_scores_topk", "mmshift_topk",
    "mmshift_gather", "mmshift_select", "mmshift_poll_status", "mmshift_status_string",
    "mmshift_last_cuda_error", "mmshift_scores_topk_noalloc",
    "mmshift_prefill_stats_workspace_size", "mmshift_prefill_stats",
    "mmshift_build_proxies_from_stats", "mmshift_select_with_stats",
    "mmshift_hidden_stats_workspace_size", "mmshift_hidden_stats",
    "mmshift_hidden_proxies_workspace_size", "mmshift_build_hidden_proxies",
    "mmshift_coverage_workspace_size", "mmshift_coverage",
    "mmshift_select_head_budgets", "mmshift_topk_head_budgets",
]
MMSHIFT_NOALLOC_SCRATCH_BYTES = 8 << 20


class Params(ctypes.Structure):
    _fields_ = [
        ("n_proxies", ctypes.c_int32), ("n_groups", ctypes.c_int32),
        ("gamma", ctypes.c_float), ("tau", ctypes.c_float), ("lambda_", ctypes.c_float),
        ("score_mode", ctypes.c_int32), ("seed", ctypes.c_uint64), ("layer_id", ctypes.c_int32),
        ("softmax_scale", ctypes.c_float), ("rope_theta", ctypes.c_float),
        ("rope_pos_offset", ctypes.c_int32),
    ]


class Shape(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("window", ctypes.c_int32), ("dtype", ctypes.c_int32),
        ("cu_seqlens", ctypes.POINTER(ctypes.c_int32)), ("budgets", ctypes.POINTER(ctypes.c_int32)),
        ("n_layers", ctypes.c_int32), ("layer_stride_kv", ctypes.c_int64),
        ("layer_stride_q", ctypes.c_int64),
    ]


MMSHIFT_N_STAGES = 8
STAGES = ("proxies", "softmax_pass", "merge", "mass_pass", "anchor_mass_sum", "cover", "topk", "gather")


class Debug(ctypes.Structure):
    _fields_ = [
        ("proxies", ctypes.c_void_p), ("group_mass", ctypes.c_void_p), ("anchor", ctypes.c_void_p),
        ("mass", ctypes.c_void_p), ("scores", ctypes.c_void_p),
        ("stage_events", ctypes.POINTER(ctypes.c_void_p)), ("n_stage_events", ctypes.c_int32),
        ("launches", ctypes.c_int32), ("score_path", ctypes.c_int32),
        ("test_stuck_wait", ctypes.c_int32),
    ]


_LIB: Optional[ctypes.CDLL] = None
_VP = ctypes.c_void_p
_SP = ctypes.POINTER(Shape)
_PP = ctypes.POINTER(Params)


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Build (if stale) and load libmmshift.so; raises if that is impossible."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if path is None:
        path = _build.build()
    if not os.path.exists(path):
        raise RuntimeError(f"libmmshift.so not found at {path}")
    lib = ctypes.CDLL(path)
    st = ctypes.c_int
    lib.mmshift_default_params.argtypes = [_PP]
    lib.mmshift_default_params.restype = None
    lib.mmshift_output_rows.argtypes = [_SP, ctypes.POINTER(ctypes.c_int64)]
    lib.mmshift_output_rows.restype = st
    lib.mmshift_workspace_size.argtypes = [_SP, _PP, ctypes.POINTER(ctypes.c_size_t)]
    lib.mmshift_workspace_size.restype = st
    lib.mmshift_build_proxies.argtypes = [_SP, _VP, _PP, _VP, _VP]
    lib.mmshift_build_proxies.restype = st
    lib.mmshift_prefill_stats_workspace_size.argtypes = [_SP, ctypes.POINTER(ctypes.c_size_t)]
    lib.mmshift_prefill_stats_workspace_size.restype = st
    lib.mmshift_prefill_stats.argtypes = [_SP, _VP, ctypes.c_int64, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_prefill_stats.restype = st
    lib.mmshift_build_proxies_from_stats.argtypes = [_SP, _VP, _PP, _VP, _VP]
    lib.mmshift_build_proxies_from_stats.restype = st
    lib.mmshift_hidden_stats_workspace_size.argtypes = [_SP, ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]
    lib.mmshift_hidden_stats_workspace_size.restype = st
    lib.mmshift_hidden_stats.argtypes = [_SP, ctypes.c_int32, _VP, ctypes.c_int64, _VP, _VP,
                                         ctypes.c_size_t, _VP]
    lib.mmshift_hidden_stats.restype = st
    lib.mmshift_hidden_proxies_workspace_size.argtypes = [_SP, ctypes.c_int32, _PP,
                                                          ctypes.POINTER(ctypes.c_size_t)]
    lib.mmshift_hidden_proxies_workspace_size.restype = st
    lib.mmshift_build_hidden_proxies.argtypes = [_SP, ctypes.c_int32, _VP, _VP, ctypes.c_int64, _VP,
                                                 _VP, _PP, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_build_hidden_proxies.restype = st
    lib.mmshift_coverage_workspace_size.argtypes = [_SP, ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]
    lib.mmshift_coverage_workspace_size.restype = st
    lib.mmshift_coverage.argtypes = [_SP, _VP, _VP, _VP, ctypes.c_int32, ctypes.c_float, _VP, _VP, _VP,
                                     ctypes.c_size_t, _VP]
    lib.mmshift_coverage.restype = st
    lib.mmshift_select_head_budgets.argtypes = [_SP, _VP, _VP, _VP, _VP, _VP, _PP, _VP, _VP, _VP, _VP,
                                                ctypes.POINTER(Debug), _VP, ctypes.c_size_t, _VP]
    lib.mmshift_select_head_budgets.restype = st
    lib.mmshift_topk_head_budgets.argtypes = [_SP, _VP, _VP, _VP, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_topk_head_budgets.restype = st
    lib.mmshift_proxy_mass.argtypes = [_SP, _VP, _VP, _VP, _PP, _VP, _VP, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_proxy_mass.restype = st
    lib.mmshift_scores_topk.argtypes = [_SP, _PP, _VP, _VP, _VP, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_scores_topk.restype = st
    lib.mmshift_topk.argtypes = [_SP, _VP, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_topk.restype = st
    lib.mmshift_gather.argtypes = [_SP, _VP, _VP, _VP, _VP, _VP, _VP, ctypes.c_size_t, _VP]
    lib.mmshift_gather.restype = st
    lib.mmshift_select.argtypes = [_SP, _VP, _VP, _VP, _VP, _PP, _VP, _VP, _VP,
                                   ctypes.POINTER(Debug), _VP, ctypes.c_size_t, _VP]
    lib.mmshift_select.restype = st
    lib.mmshift_select_with_stats.argtypes = [_SP, _VP, _VP, _VP, _VP, _PP, _VP, _VP, _VP,
                                              ctypes.POINTER(Debug), _VP, ctypes.c_size_t, _VP]
    lib.mmshift_select_with_stats.restype = st
    lib.mmshift_scores_topk_noalloc.argtypes = [_SP, _PP, _VP, _VP, _VP, _VP, _VP]
    lib.mmshift_scores_topk_noalloc.restype = st
    lib.mmshift_poll_status.argtypes = [_VP, _VP]
    lib.mmshift_poll_status.restype = st
    lib.mmshift_status_string.argtypes = [st]
    lib.mmshift_status_string.restype = ctypes.c_char_p
    lib.mmshift_last_cuda_error.argtypes = []
    lib.mmshift_last_cuda_error.restype = ctypes.c_char_p
    _LIB = lib
    return lib


class MMShiftError(RuntimeError):
    def __init__(self, code: int, where: str):
        lib = load_library()
        msg = lib.mmshift_status_string(code).decode()
        if code == MMSHIFT_ERR_CUDA:
            msg += ": " + lib.mmshift_last_cuda_error().decode()
        super().__init__(f"{where}: {msg} (status {code})")
        self.code = code


def check(code: int, where: str) -> None:
    if code != MMSHIFT_OK:
        raise MMShiftError(code, where)


def make_shape(n_q_heads: int, n_kv_heads: int, head_dim: int, window: int, dtype: int,
               cu_seqlens: Sequence[int], budgets: Sequence[int], n_layers: int = 1,
               layer_stride_kv: int = 0, layer_stride_q: int = 0) -> Shape:
    """Shape with its host arrays kept alive on the returned object."""
    cu = (ctypes.c_int32 * len(cu_seqlens))(*[int(x) for x in cu_seqlens])
    bu = (ctypes.c_int32 * len(budgets))(*[int(x) for x in budgets])
    s = Shape(batch=len(budgets), n_q_heads=n_q_heads, n_kv_heads=n_kv_heads, head_dim=head_dim,
              window=window, dtype=dtype, cu_seqlens=cu, budgets=bu, n_layers=n_layers,
              layer_stride_kv=layer_stride_kv, layer_stride_q=layer_stride_q)
    s._keep = (cu, bu)
    return s


def default_params(**kw) -> Params:
    p = Params()
    load_library().mmshift_default_params(ctypes.byref(p))
    for k, v in kw.items():
        setattr(p, "lambda_" if k in ("lam", "lambda") else k, v)
    return p


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "cuda_stream"):          # torch.cuda.Stream
        return x.cuda_stream
    return x.data_ptr()


def mmshift_output_rows(shape: Shape) -> int:
    r = ctypes.c_int64()
    check(load_library().mmshift_output_rows(ctypes.byref(shape), ctypes.byref(r)), "mmshift_output_rows")
    return r.value


def mmshift_workspace_size(shape: Shape, params: Optional[Params]) -> int:
    n = ctypes.c_size_t()
    pp = ctypes.byref(params) if params is not None else None
    check(load_library().mmshift_workspace_size(ctypes.byref(shape), pp, ctypes.byref(n)),
          "mmshift_workspace_size")
    return n.value


def mmshift_build_proxies(shape, qwin, params, proxies, stream=None) -> int:
    return load_library().mmshift_build_proxies(ctypes.byref(shape), _ptr(qwin), ctypes.byref(params),
                                                _ptr(proxies), _ptr(stream))


def mmshift_prefill_stats_workspace_size(shape: Shape) -> int:
    n = ctypes.c_size_t()
    check(load_library().mmshift_prefill_stats_workspace_size(ctypes.byref(shape), ctypes.byref(n)),
          "mmshift_prefill_stats_workspace_size")
    return n.value


def mmshift_prefill_stats(shape, qfull, qfull_layer_stride, stats, workspace, workspace_bytes,
                          stream=None) -> int:
    return load_library().mmshift_prefill_stats(ctypes.byref(shape), _ptr(qfull),
                                                int(qfull_layer_stride), _ptr(stats),
                                                _ptr(workspace), workspace_bytes, _ptr(stream))



def mmshift_hidden_stats_workspace_size(shape: Shape, d_model: int) -> int:
    n = ctypes.c_size_t()
    check(load_library().mmshift_hidden_stats_workspace_size(ctypes.byref(shape), int(d_model),
                                                             ctypes.byref(n)),
          "mmshift_hidden_stats_workspace_size")
    return n.value


def mmshift_hidden_stats(shape, d_model, H, h_layer_stride, stats, workspace, workspace_bytes,
                         stream=None) -> int:
    return load_library().mmshift_hidden_stats(ctypes.byref(shape), int(d_model), _ptr(H),
                                               int(h_layer_stride), _ptr(stats), _ptr(workspace),
                                               workspace_bytes, _ptr(stream))


def mmshift_hidden_proxies_workspace_size(shape: Shape, d_model: int, params) -> int:
    n = ctypes.c_size_t()
    check(load_library().mmshift_hidden_proxies_workspace_size(ctypes.byref(shape), int(d_model),
                                                               ctypes.byref(params), ctypes.byref(n)),
          "mmshift_hidden_proxies_workspace_size")
    return n.value


def mmshift_build_hidden_proxies(shape, d_model, hstats, W_Q, wq_layer_stride, bias_q, rope_pos,
                                 params, proxies, workspace, workspace_bytes, stream=None) -> int:
    """rope_pos: None or a sequence of per-request positions (host int32)."""
    pos = None
    if rope_pos is not None:
        pos = (ctypes.c_int32 * len(rope_pos))(*[int(x) for x in rope_pos])
    return load_library().mmshift_build_hidden_proxies(
        ctypes.byref(shape), int(d_model), _ptr(hstats), _ptr(W_Q), int(wq_layer_stride),
        _ptr(bias_q), pos, ctypes.byref(params), _ptr(proxies), _ptr(workspace), workspace_bytes,
        _ptr(stream))


def mmshift_build_proxies_from_stats(shape, stats, params, proxies, stream=None) -> int:
    return load_library().mmshift_build_proxies_from_stats(ctypes.byref(shape), _ptr(stats),
                                                           ctypes.byref(params), _ptr(proxies),
                                                           _ptr(stream))


def mmshift_proxy_mass(shape, K, qwin, proxies, params, group_mass, anchor, mass, workspace,
                       workspace_bytes, stream=None) -> int:
    return load_library().mmshift_proxy_mass(
        ctypes.byref(shape), _ptr(K), _ptr(qwin), _ptr(proxies), ctypes.byref(params),
        _ptr(group_mass), _ptr(anchor), _ptr(mass), _ptr(workspace), workspace_bytes, _ptr(stream))


def mmshift_scores_topk(shape, params, group_mass, anchor, scores, out_idx, workspace,
                        workspace_bytes, stream=None) -> int:
    return load_library().mmshift_scores_topk(
        ctypes.byref(shape), ctypes.byref(params), _ptr(group_mass), _ptr(anchor), _ptr(scores),
        _ptr(out_idx), _ptr(workspace), workspace_bytes, _ptr(stream))


def mmshift_scores_topk_noalloc(shape, params, group_mass, anchor, scores, out_idx,
                                stream=None) -> int:
    """Allocation-free vote + top-k: scratch comes from a static device array
    inside the library (for callers that cannot allocate device memory)."""
    return load_library().mmshift_scores_topk_noalloc(
        ctypes.byref(shape), ctypes.byref(params), _ptr(group_mass), _ptr(anchor), _ptr(scores),
        _ptr(out_idx), _ptr(stream))


def mmshift_topk(shape, scores, out_idx, workspace, workspace_bytes, stream=None) -> int:
    return load_library().mmshift_topk(ctypes.byref(shape), _ptr(scores), _ptr(out_idx),
                                       _ptr(workspace), workspace_bytes, _ptr(stream))


def mmshift_gather(shape, K, V, idx, out_K, out_V, workspace, workspace_bytes, stream=None) -> int:
    return load_library().mmshift_gather(ctypes.byref(shape), _ptr(K), _ptr(V), _ptr(idx),
                                         _ptr(out_K), _ptr(out_V), _ptr(workspace), workspace_bytes,
                                         _ptr(stream))


def mmshift_select(shape, K, V, qwin, proxies_in, params, out_idx, out_K, out_V, debug,
                   workspace, workspace_bytes, stream=None) -> int:
    dbg = ctypes.byref(debug) if debug is not None else None
    return load_library().mmshift_select(
        ctypes.byref(shape), _ptr(K), _ptr(V), _ptr(qwin), _ptr(proxies_in), ctypes.byref(params),
        _ptr(out_idx), _ptr(out_K), _ptr(out_V), dbg, _ptr(workspace), workspace_bytes, _ptr(stream))



def mmshift_select_with_stats(shape, K, V, qwin, stats, params, out_idx, out_K, out_V, debug,
                              workspace, workspace_bytes, stream=None) -> int:
    dbg = ctypes.byref(debug) if debug is not None else None
    return load_library().mmshift_select_with_stats(
        ctypes.byref(shape), _ptr(K), _ptr(V), _ptr(qwin), _ptr(stats), ctypes.byref(params),
        _ptr(out_idx), _ptr(out_K), _ptr(out_V), dbg, _ptr(workspace), workspace_bytes, _ptr(stream))



def mmshift_coverage_workspace_size(shape: Shape, n_dec: int) -> int:
    n = ctypes.c_size_t()
    check(load_library().mmshift_coverage_workspace_size(ctypes.byref(shape), int(n_dec),
                                                         ctypes.byref(n)),
          "mmshift_coverage_workspace_size")
    return n.value


def mmshift_coverage(shape, K, qwin, dec_q, n_dec, softmax_scale, idx, cov, workspace,
                     workspace_bytes, stream=None) -> int:
    return load_library().mmshift_coverage(ctypes.byref(shape), _ptr(K), _ptr(qwin), _ptr(dec_q),
                                           int(n_dec), float(softmax_scale), _ptr(idx), _ptr(cov),
                                           _ptr(workspace), workspace_bytes, _ptr(stream))



def mmshift_select_head_budgets(shape, K, V, qwin, proxies_in, head_budgets, params, out_idx,
                                out_count, out_K, out_V, debug, workspace, workspace_bytes,
                                stream=None) -> int:
    dbg = ctypes.byref(debug) if debug is not None else None
    return load_library().mmshift_select_head_budgets(
        ctypes.byref(shape), _ptr(K), _ptr(V), _ptr(qwin), _ptr(proxies_in), _ptr(head_budgets),
        ctypes.byref(params), _ptr(out_idx), _ptr(out_count), _ptr(out_K), _ptr(out_V), dbg,
        _ptr(workspace), workspace_bytes, _ptr(stream))


def mmshift_topk_head_budgets(shape, scores, head_budgets, out_idx, out_count, workspace,
                              workspace_bytes, stream=None) -> int:
    return load_library().mmshift_topk_head_budgets(
        ctypes.byref(shape), _ptr(scores), _ptr(head_budgets), _ptr(out_idx), _ptr(out_count),
        _ptr(workspace), workspace_bytes, _ptr(stream))


def mmshift_poll_status(workspace, stream=None) -> int:
    return load_library().mmshift_poll_status(_ptr(workspace), _ptr(stream))


def make_debug(proxies=None, group_mass=None, anchor=None, mass=None, scores=None,
               stage_events=None, test_stuck_wait=0) -> Debug:
    """stage_events: sequence of MMSHIFT_N_STAGES + 1 torch.cuda.Event (timing).
    test_stuck_wait: test of the bounded device waits (see mmshift.h)."""
    dbg = Debug(proxies=_ptr(proxies), group_mass=_ptr(group_mass), anchor=_ptr(anchor),
                mass=_ptr(mass), scores=_ptr(scores), test_stuck_wait=int(test_stuck_wait))
    if stage_events is not None:
        arr = (ctypes.c_void_p * len(stage_events))(*[e.cuda_event for e in stage_events])
        dbg.stage_events = arr
        dbg.n_stage_events = len(stage_events)
        dbg._keep = arr
    return dbg
