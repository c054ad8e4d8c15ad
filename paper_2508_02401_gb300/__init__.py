"""Python binding of libckv (include/ckv.h): CompressKV's prefill-time KV-cache compression
step on GB300.

The functions here carry the C names and only marshal arguments (torch tensors -> device
pointers, numpy arrays -> host pointers, the current torch stream -> cudaStream_t).  Every step
of the computation runs in the library's CUDA kernels; there is no other implementation behind
these calls.  Loading fails loudly if the library has not been built.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass

import numpy as np

__all__ = [
    "CkvError", "Config", "Batch", "lib_path", "load",
    "ckv_workspace_size", "ckv_keep_lengths", "ckv_score_window", "ckv_pool", "ckv_select_topk",
    "ckv_gather_compact", "ckv_select_compact", "ckv_compress_layer", "ckv_read_device_status",
    "ckv_status_string",
    "ckv_abi_version", "ckv_score_window_static", "POOL_MAX", "POOL_AVG", "POOL_THEN_SUM", "SUM_THEN_POOL",
    "SCOPE_KV_HEAD", "SCOPE_LAYER", "ckv_layer_error_scores", "ckv_allocate_budgets",
    "SCORE_AUTO", "SCORE_RESIDENT", "SCORE_RELOAD", "ckv_score_window_lse",
    "ckv_compress_layer_lse", "ckv_semantic_retrieval_scores", "ckv_set_wait_limit_us",
    "new_workspace", "new_outputs", "LayerIO", "ckv_workspace_size_layers", "ckv_score_windows",
    "ckv_compress_layers", "ckv_compress_layers_lse", "new_layers_workspace", "ckv_score_windows_lse",
]

POOL_MAX, POOL_AVG = 0, 1
SCOPE_KV_HEAD, SCOPE_LAYER = 0, 1
POOL_THEN_SUM, SUM_THEN_POOL = 0, 1
SCORE_AUTO, SCORE_RESIDENT, SCORE_RELOAD = 0, 1, 2
_HERE = os.path.dirname(os.path.abspath(__file__))
_lib = None


def lib_path() -> str:
    return os.path.join(_HERE, "libckv.so")


class CkvError(RuntimeError):
    def __init__(self, status: int, where: str, message: str):
        self.status = status
        super().__init__(f"{where}: {_STATUS.get(status, status)}: {message}")


_STATUS = {0: "CKV_OK", 1: "CKV_ERR_INVALID_ARG", 2: "CKV_ERR_UNSUPPORTED", 3: "CKV_ERR_WORKSPACE",
           4: "CKV_ERR_CUDA", 5: "CKV_ERR_DEVICE"}


class _Config(C.Structure):
    _fields_ = [("num_layers", C.c_int32), ("num_q_heads", C.c_int32), ("num_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("window", C.c_int32), ("pool_kernel", C.c_int32),
                ("pool_type", C.c_int32), ("head_order", C.c_int32), ("scope", C.c_int32),
                ("softmax_scale", C.c_float),
                ("max_ctas", C.c_int32), ("score_path", C.c_int32), ("head_mask", C.c_void_p),
                ("budgets", C.c_void_p)]


class _LayerIO(C.Structure):
    _fields_ = [("layer", C.c_int32), ("q_win", C.c_void_p), ("k", C.c_void_p), ("v", C.c_void_p),
                ("tok_stride", C.c_int64), ("head_stride", C.c_int64), ("scores", C.c_void_p),
                ("idx", C.c_void_p), ("cu_keep_dev", C.c_void_p), ("k_out", C.c_void_p),
                ("v_out", C.c_void_p), ("pooled_out", C.c_void_p), ("lse", C.c_void_p),
                ("lse_head_stride", C.c_int64)]


class _Batch(C.Structure):
    _fields_ = [("num_seqs", C.c_int32), ("cu_seqlens_host", C.c_void_p),
                ("cu_seqlens_dev", C.c_void_p)]


def load():
    """Loads libckv.so (built by ``paper_2508_02401_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    path = lib_path()
    if not os.path.exists(path):
        raise ImportError(f"libckv.so is not built ({path}); run "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = C.CDLL(path)
    P, I32, I64, SZ = C.c_void_p, C.c_int32, C.c_int64, C.c_size_t
    cfg, bat = C.POINTER(_Config), C.POINTER(_Batch)
    sigs = {
        "ckv_abi_version": ([], I32),
        "ckv_status_string": ([C.c_int], C.c_char_p),
        "ckv_last_error_message": ([], C.c_char_p),
        "ckv_workspace_size": ([cfg, I32, bat, C.POINTER(SZ)], C.c_int),
        "ckv_keep_lengths": ([cfg, I32, bat, P, C.POINTER(I32)], C.c_int),
        "ckv_score_window": ([cfg, I32, bat, P, P, I64, I64, P, P, SZ, P], C.c_int),
        "ckv_pool": ([cfg, I32, bat, P, P, P], C.c_int),
        "ckv_select_topk": ([cfg, I32, bat, P, P, P, P, SZ, P], C.c_int),
        "ckv_gather_compact": ([cfg, bat, I32, P, P, I64, I64, P, P, P, P, P, SZ, P], C.c_int),
        "ckv_select_compact": ([cfg, I32, bat, P, P, P, I64, I64, P, P, P, P, P, P, SZ, P], C.c_int),
        "ckv_compress_layer": ([cfg, I32, bat, P, P, P, I64, I64, P, P, P, P, P, P, SZ, P], C.c_int),
        "ckv_read_device_status": ([P, P, I32, C.POINTER(I32), C.POINTER(I32)], C.c_int),
        "ckv_score_window_static": ([cfg, I32, bat, P, P, I64, I64, P, P, P], C.c_int),
        "ckv_score_window_lse": ([cfg, I32, bat, P, P, I64, I64, P, I64, P, P, SZ, P], C.c_int),
        "ckv_semantic_retrieval_scores": ([cfg, I32, bat, P, P, I64, I64, P, I64, P, P, P, P, SZ, P],
                                          C.c_int),
        "ckv_compress_layer_lse": ([cfg, I32, bat, P, P, P, I64, I64, P, I64, P, P, P, P, P, P, SZ, P],
                                   C.c_int),
        "ckv_layer_error_scores": ([P, I32, I32, P], C.c_int),
        "ckv_set_wait_limit_us": ([C.c_uint32], C.c_int),
        "ckv_allocate_budgets": ([P, I32, I64, I32, I32, P], C.c_int),
        "ckv_workspace_size_layers": ([cfg, I32, P, bat, C.POINTER(SZ)], C.c_int),
        "ckv_score_windows": ([cfg, I32, P, bat, P, SZ, P], C.c_int),
        "ckv_score_windows_lse": ([cfg, I32, P, bat, P, SZ, P], C.c_int),
        "ckv_compress_layers": ([cfg, I32, P, bat, P, SZ, P], C.c_int),
        "ckv_compress_layers_lse": ([cfg, I32, P, bat, P, SZ, P], C.c_int),
    }
    for name, (args, res) in sigs.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def _check(rc: int, where: str):
    if rc != 0:
        raise CkvError(rc, where, load().ckv_last_error_message().decode())


@dataclass
class Config:
    """Per-model settings: the paper's per-layer head mask and per-layer budgets."""
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    window: int
    pool_kernel: int
    pool_type: int
    head_order: int
    head_mask: np.ndarray   # uint8 [num_layers, num_q_heads]
    budgets: np.ndarray     # int32 [num_layers]
    softmax_scale: float = 0.0
    head_dim: int = 128
    max_ctas: int = 0       # SMs one call's scoring kernel may occupy (0 = all)
    scope: int = SCOPE_KV_HEAD  # SCOPE_LAYER: one selection per sequence for all KV heads
    score_path: int = 0     # SCORE_AUTO / SCORE_RESIDENT / SCORE_RELOAD (the scoring kernel)

    def __post_init__(self):
        self.head_mask = np.ascontiguousarray(self.head_mask, dtype=np.uint8)
        self.budgets = np.ascontiguousarray(self.budgets, dtype=np.int32)
        self._c = _Config(self.num_layers, self.num_q_heads, self.num_kv_heads, self.head_dim,
                          self.window, self.pool_kernel, self.pool_type, self.head_order,
                          self.scope, self.softmax_scale, self.max_ctas, self.score_path,
                          self.head_mask.ctypes.data, self.budgets.ctypes.data)

    @classmethod
    def from_workload(cls, wl, **overrides):
        kw = dict(num_layers=wl.num_layers, num_q_heads=wl.num_q_heads,
                  num_kv_heads=wl.num_kv_heads, window=wl.window, pool_kernel=wl.pool_kernel,
                  pool_type=POOL_MAX if wl.pool_type == "max" else POOL_AVG,
                  head_order=POOL_THEN_SUM if wl.head_order == "pool_then_sum" else SUM_THEN_POOL,
                  head_mask=wl.head_mask(), budgets=wl.budgets(), head_dim=wl.head_dim,
                  scope=SCOPE_LAYER if getattr(wl, "scope", "kv_head") == "layer" else SCOPE_KV_HEAD)
        kw.update(overrides)
        return cls(**kw)

    @property
    def num_vectors(self) -> int:
        """Selections per sequence: the rows of the pooled scores."""
        return 1 if self.scope == SCOPE_LAYER else self.num_kv_heads

    @property
    def ref(self):
        return C.byref(self._c)


class Batch:
    """A varlen batch: host and device copies of cu_seqlens [S+1]."""

    def __init__(self, cu_seqlens, device=None, cu_seqlens_dev=None):
        import torch
        self.cu_host = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
        if cu_seqlens_dev is None:
            cu_seqlens_dev = torch.from_numpy(self.cu_host.copy()).to(device or "cuda")
        self.cu_dev = cu_seqlens_dev
        self._c = _Batch(len(self.cu_host) - 1, self.cu_host.ctypes.data, self.cu_dev.data_ptr())

    @property
    def num_seqs(self) -> int:
        return len(self.cu_host) - 1

    @property
    def total_tokens(self) -> int:
        return int(self.cu_host[-1])

    @property
    def ref(self):
        return C.byref(self._c)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream if isinstance(stream, int) else stream.cuda_stream)


def ckv_abi_version() -> int:
    return load().ckv_abi_version()


def ckv_status_string(status: int) -> str:
    return load().ckv_status_string(status).decode()


def ckv_workspace_size(cfg: Config, layer: int, batch: Batch) -> int:
    n = C.c_size_t(0)
    _check(load().ckv_workspace_size(cfg.ref, layer, batch.ref, C.byref(n)), "ckv_workspace_size")
    return n.value


def ckv_keep_lengths(cfg: Config, layer: int, batch: Batch):
    """Returns (cu_keep [S+1] int32 numpy, n_sel)."""
    out = np.zeros(batch.num_seqs + 1, np.int32)
    n_sel = C.c_int32(0)
    _check(load().ckv_keep_lengths(cfg.ref, layer, batch.ref, out.ctypes.data, C.byref(n_sel)),
           "ckv_keep_lengths")
    return out, n_sel.value


def ckv_layer_error_scores(errors) -> np.ndarray:
    """Eq. 11-13: per-layer scores (float64 [L]) from errors [datasets, L] (host)."""
    e = np.ascontiguousarray(errors, dtype=np.float64)
    if e.ndim != 2:
        raise ValueError("errors must be [datasets, layers]")
    out = np.zeros(e.shape[1], np.float64)
    _check(load().ckv_layer_error_scores(e.ctypes.data, e.shape[0], e.shape[1], out.ctypes.data),
           "ckv_layer_error_scores")
    return out


def ckv_allocate_budgets(scores, total_budget: int, min_budget: int = 32, max_budget: int | None = None):
    """Algorithm 1: int32 [L] budgets; max_budget defaults to 3 * total_budget // L."""
    s = np.ascontiguousarray(scores, dtype=np.float64)
    L = s.shape[0]
    if max_budget is None:
        max_budget = 3 * int(total_budget) // max(L, 1)
    out = np.zeros(L, np.int32)
    _check(load().ckv_allocate_budgets(s.ctypes.data, L, int(total_budget), int(min_budget),
                                       int(max_budget), out.ctypes.data), "ckv_allocate_budgets")
    return out


def ckv_set_wait_limit_us(microseconds: int):
    """Limit of the kernels' bounded waits for later calls (0 = the default, about 2 s)."""
    _check(load().ckv_set_wait_limit_us(int(microseconds)), "ckv_set_wait_limit_us")


def ckv_score_window(cfg, layer, batch, q_win, k, scores, workspace, stream=None,
                     tok_stride=0, head_stride=0):
    _check(load().ckv_score_window(cfg.ref, layer, batch.ref, _ptr(q_win), _ptr(k), tok_stride,
                                   head_stride, _ptr(scores), _ptr(workspace),
                                   workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_score_window")


def ckv_pool(cfg, layer, batch, scores, pooled, stream=None):
    _check(load().ckv_pool(cfg.ref, layer, batch.ref, _ptr(scores), _ptr(pooled), _stream(stream)),
           "ckv_pool")


def ckv_select_topk(cfg, layer, batch, pooled, idx, cu_keep_dev, workspace, stream=None):
    _check(load().ckv_select_topk(cfg.ref, layer, batch.ref, _ptr(pooled), _ptr(idx),
                                  _ptr(cu_keep_dev), _ptr(workspace),
                                  workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_select_topk")


def ckv_gather_compact(cfg, batch, t_keep, k, v, idx, cu_keep_dev, k_out, v_out, workspace,
                       stream=None, tok_stride=0, head_stride=0):
    _check(load().ckv_gather_compact(cfg.ref, batch.ref, t_keep, _ptr(k), _ptr(v), tok_stride,
                                     head_stride, _ptr(idx), _ptr(cu_keep_dev), _ptr(k_out),
                                     _ptr(v_out), _ptr(workspace),
                                     workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_gather_compact")


def ckv_select_compact(cfg, layer, batch, scores, k, v, idx, cu_keep_dev, k_out, v_out, workspace,
                       pooled_out=None, stream=None, tok_stride=0, head_stride=0):
    """Pool, top-k, compaction and gather of one layer from ckv_score_window's scores."""
    _check(load().ckv_select_compact(cfg.ref, layer, batch.ref, _ptr(scores), _ptr(k), _ptr(v),
                                     tok_stride, head_stride, _ptr(idx), _ptr(cu_keep_dev),
                                     _ptr(k_out), _ptr(v_out), _ptr(pooled_out), _ptr(workspace),
                                     workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_select_compact")


def ckv_compress_layer(cfg, layer, batch, q_win, k, v, idx, cu_keep_dev, k_out, v_out, workspace,
                       pooled_out=None, stream=None, tok_stride=0, head_stride=0):
    _check(load().ckv_compress_layer(cfg.ref, layer, batch.ref, _ptr(q_win), _ptr(k), _ptr(v),
                                     tok_stride, head_stride, _ptr(idx), _ptr(cu_keep_dev),
                                     _ptr(k_out), _ptr(v_out), _ptr(pooled_out), _ptr(workspace),
                                     workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_compress_layer")


def ckv_score_window_lse(cfg, layer, batch, q_win, k, lse, scores, workspace, lse_head_stride=0,
                         stream=None, tok_stride=0, head_stride=0):
    """ckv_score_window with the window rows' lse given: lse [H_q, >= S*w] fp32 natural log."""
    _check(load().ckv_score_window_lse(cfg.ref, layer, batch.ref, _ptr(q_win), _ptr(k), tok_stride,
                                       head_stride, _ptr(lse), lse_head_stride, _ptr(scores),
                                       _ptr(workspace), workspace.numel() * workspace.element_size(),
                                       _stream(stream)), "ckv_score_window_lse")


def ckv_compress_layer_lse(cfg, layer, batch, q_win, k, v, lse, idx, cu_keep_dev, k_out, v_out,
                           workspace, lse_head_stride=0, pooled_out=None, stream=None, tok_stride=0,
                           head_stride=0):
    """ckv_compress_layer with the window rows' lse given (layout as ckv_score_window_lse)."""
    _check(load().ckv_compress_layer_lse(cfg.ref, layer, batch.ref, _ptr(q_win), _ptr(k), _ptr(v),
                                         tok_stride, head_stride, _ptr(lse), lse_head_stride,
                                         _ptr(idx), _ptr(cu_keep_dev), _ptr(k_out), _ptr(v_out),
                                         _ptr(pooled_out), _ptr(workspace),
                                         workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_compress_layer_lse")


def ckv_semantic_retrieval_scores(cfg, layer, batch, q_dec, k, lse, in_answer, span, srs, workspace,
                                  lse_head_stride=0, stream=None, tok_stride=0, head_stride=0):
    """Eq. 5: srs [H_q] += the selected heads' attention of the in-answer decode steps on the
    answer span.  q_dec like q_win (w = cfg.window decode steps), k = context + generated keys,
    lse [H_q, >= S*w], in_answer uint8 [S*w], span int32 [S, 2] (all device tensors)."""
    _check(load().ckv_semantic_retrieval_scores(
        cfg.ref, layer, batch.ref, _ptr(q_dec), _ptr(k), tok_stride, head_stride, _ptr(lse),
        lse_head_stride, _ptr(in_answer), _ptr(span), _ptr(srs), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)), "ckv_semantic_retrieval_scores")


def ckv_score_window_static(cfg, layer, batch, q_win, k, scores, status_out=None, stream=None,
                            tok_stride=0, head_stride=0):
    """ckv_score_window without a workspace: the library's fixed static scratch is used."""
    _check(load().ckv_score_window_static(cfg.ref, layer, batch.ref, _ptr(q_win), _ptr(k),
                                          tok_stride, head_stride, _ptr(scores), _ptr(status_out),
                                          _stream(stream)), "ckv_score_window_static")


@dataclass
class LayerIO:
    """One layer of a multi-layer call (ckv_layer_io): the layer index and its tensors."""
    layer: int
    q_win: object
    k: object
    v: object = None
    scores: object = None       # ckv_score_windows
    idx: object = None          # ckv_compress_layers
    cu_keep_dev: object = None
    k_out: object = None
    v_out: object = None
    pooled_out: object = None
    tok_stride: int = 0
    head_stride: int = 0
    lse: object = None          # the _lse calls: [H_q, S*w] fp32
    lse_head_stride: int = 0


def _layer_ios(ios):
    arr = (_LayerIO * len(ios))()
    for i, x in enumerate(ios):
        arr[i] = _LayerIO(x.layer, *(None if t is None else t.data_ptr() for t in (x.q_win, x.k, x.v)),
                          x.tok_stride, x.head_stride,
                          *(None if t is None else t.data_ptr()
                            for t in (x.scores, x.idx, x.cu_keep_dev, x.k_out, x.v_out, x.pooled_out,
                                      x.lse)),
                          x.lse_head_stride)
    return arr


def ckv_workspace_size_layers(cfg, ios, batch) -> int:
    n = C.c_size_t(0)
    arr = _layer_ios(ios)
    _check(load().ckv_workspace_size_layers(cfg.ref, len(ios), arr, batch.ref, C.byref(n)),
           "ckv_workspace_size_layers")
    return n.value


def new_layers_workspace(cfg, ios, batch, device="cuda"):
    """A zeroed workspace of ckv_workspace_size_layers bytes (uint8 tensor)."""
    import torch
    return torch.zeros(ckv_workspace_size_layers(cfg, ios, batch), dtype=torch.uint8, device=device)


def ckv_score_windows(cfg, ios, batch, workspace, stream=None):
    """ckv_score_window for every LayerIO of `ios` (their `scores`), in one persistent launch."""
    arr = _layer_ios(ios)
    _check(load().ckv_score_windows(cfg.ref, len(ios), arr, batch.ref, _ptr(workspace),
                                    workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_score_windows")


def ckv_score_windows_lse(cfg, ios, batch, workspace, stream=None):
    """ckv_score_window_lse for every LayerIO of `ios` (their `scores`, each with its `lse`), in
    one persistent single-pass launch."""
    arr = _layer_ios(ios)
    _check(load().ckv_score_windows_lse(cfg.ref, len(ios), arr, batch.ref, _ptr(workspace),
                                        workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_score_windows_lse")


def ckv_compress_layers(cfg, ios, batch, workspace, stream=None):
    """ckv_compress_layer for every LayerIO of `ios`: one scoring launch, then the selections."""
    arr = _layer_ios(ios)
    _check(load().ckv_compress_layers(cfg.ref, len(ios), arr, batch.ref, _ptr(workspace),
                                      workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_compress_layers")


def ckv_compress_layers_lse(cfg, ios, batch, workspace, stream=None):
    """ckv_compress_layer_lse for every LayerIO of `ios` (each with its `lse`): one single-pass
    scoring launch over every layer, then the selections in one launch."""
    arr = _layer_ios(ios)
    _check(load().ckv_compress_layers_lse(cfg.ref, len(ios), arr, batch.ref, _ptr(workspace),
                                          workspace.numel() * workspace.element_size(), _stream(stream)),
           "ckv_compress_layers_lse")


def ckv_read_device_status(workspace, stream=None, reset=True):
    """Synchronises the stream; returns (code, detail) of the workspace status word."""
    code, detail = C.c_int32(0), C.c_int32(0)
    _check(load().ckv_read_device_status(_ptr(workspace), _stream(stream), 1 if reset else 0,
                                         C.byref(code), C.byref(detail)), "ckv_read_device_status")
    return code.value, detail.value


def new_workspace(cfg, layer, batch, device="cuda"):
    """A zeroed workspace of ckv_workspace_size bytes (uint8 tensor, 256-byte aligned)."""
    import torch
    n = ckv_workspace_size(cfg, layer, batch)
    return torch.zeros(n, dtype=torch.uint8, device=device)


def new_outputs(cfg, layer, batch, device="cuda"):
    """Allocates (idx, cu_keep_dev, k_out, v_out) for one layer; returns them with cu_keep_host."""
    import torch
    cu_keep, _ = ckv_keep_lengths(cfg, layer, batch)
    tk = int(cu_keep[-1])
    idx = torch.empty((cfg.num_kv_heads, tk), dtype=torch.int32, device=device)
    cu_keep_dev = torch.empty(batch.num_seqs + 1, dtype=torch.int32, device=device)
    k_out = torch.empty((tk, cfg.num_kv_heads, cfg.head_dim), dtype=torch.bfloat16, device=device)
    v_out = torch.empty_like(k_out)
    return idx, cu_keep_dev, k_out, v_out, cu_keep
