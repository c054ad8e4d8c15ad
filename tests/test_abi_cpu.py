"""The C ABI without a GPU: the library builds, loads, exports every declared symbol, and
rejects bad arguments on the host before anything would be enqueued."""
import ctypes as C
import os
import re
import subprocess

import numpy as np
import pytest

import paper_2508_02401_gb300 as ckv
from paper_2508_02401_gb300 import build as ckv_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ckv.h")


@pytest.fixture(scope="module")
def lib():
    ckv_build.build()
    return ckv.load()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ckv_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("ckv_score_window", "ckv_pool", "ckv_select_topk", "ckv_gather_compact",
              "ckv_compress_layer", "ckv_workspace_size", "ckv_keep_lengths", "ckv_score_windows",
              "ckv_compress_layers", "ckv_compress_layers_lse", "ckv_workspace_size_layers",
              "ckv_score_windows_lse",
              "ckv_read_device_status", "ckv_status_string"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", ckv.lib_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (ckv_\w+)", out))
    missing = [n for n in _declared() if n not in exported]
    assert not missing, missing
    assert all(not n.startswith("_Z") for n in exported)  # plain C names
    for n in _declared():
        assert hasattr(lib, n)


def test_version_and_status_strings(lib):
    assert ckv.ckv_abi_version() == 7
    assert ckv.ckv_status_string(0) == "CKV_OK"
    assert ckv.ckv_status_string(3) == "CKV_ERR_WORKSPACE"


def _cfg(**kw):
    base = dict(num_layers=2, num_q_heads=32, num_kv_heads=8, window=32, pool_kernel=7,
                pool_type=0, head_order=0, head_mask=np.tile(np.eye(4, dtype=np.uint8)[0], (2, 8)),
                budgets=np.array([128, 64], np.int32))
    base.update(kw)
    return ckv.Config(**base)


class FakeBatch:
    """A batch whose device pointer is never dereferenced (host validation only)."""

    def __init__(self, cu):
        self.cu_host = np.ascontiguousarray(cu, np.int32)
        self._c = ckv._Batch(len(cu) - 1, self.cu_host.ctypes.data, 0x10000)

    num_seqs = property(lambda self: len(self.cu_host) - 1)
    ref = property(lambda self: C.byref(self._c))


def test_workspace_and_keep_lengths(lib):
    cfg = _cfg()
    b = FakeBatch([0, 2048, 2100, 2110])
    cu_keep, n_sel = ckv.ckv_keep_lengths(cfg, 0, b)
    assert list(cu_keep) == [0, 128, 180, 190] and n_sel == 8
    cu_keep, _ = ckv.ckv_keep_lengths(cfg, 1, b)
    assert list(cu_keep) == [0, 64, 116, 126]
    n = ckv.ckv_workspace_size(cfg, 0, b)
    assert n % 256 == 0 and n >= 8 * 2110 * 4 + 8 * 2110 * 4


_P = 0x20000  # a 256-byte-aligned fake device address


def _call_compress(lib, cfg, batch, layer=0, q=_P, k=_P, v=_P, ws=_P, ws_bytes=1 << 30,
                   tok=0, head=0, idx=_P, cu_keep=_P):
    return lib.ckv_compress_layer(cfg.ref, layer, batch.ref, q, k, v, tok, head, idx, cu_keep, _P,
                                  _P, None, ws, ws_bytes, None)


@pytest.mark.parametrize("change,expect", [
    (dict(head_dim=64), 2), (dict(head_dim=0), 1), (dict(window=0), 1), (dict(window=65), 2),
    (dict(pool_kernel=4), 1), (dict(pool_kernel=0), 1), (dict(pool_kernel=65), 2),
    (dict(pool_type=2), 1), (dict(head_order=5), 1), (dict(num_kv_heads=5), 1),
    (dict(softmax_scale=-1.0), 1), (dict(softmax_scale=float("nan")), 1),
    (dict(budgets=np.array([16, 64], np.int32)), 1),              # budget below the window
    (dict(head_mask=np.zeros((2, 32), np.uint8)), 1),             # group without a head
    (dict(num_q_heads=512, num_kv_heads=8, head_mask=np.ones((2, 512), np.uint8)), 2),
    (dict(scope=2), 1),
    (dict(score_path=3), 1),
    (dict(score_path=-1), 1),
    (dict(scope=1, head_mask=np.zeros((2, 32), np.uint8)), 1),    # layer without a head
])
def test_config_errors(lib, change, expect):
    cfg = _cfg(**change)
    rc = _call_compress(lib, cfg, FakeBatch([0, 4096]))
    assert rc == expect, lib.ckv_last_error_message()


def test_argument_errors(lib):
    cfg, b = _cfg(), FakeBatch([0, 4096, 5000])
    assert _call_compress(lib, cfg, b, layer=2) == 1
    assert _call_compress(lib, cfg, b, layer=-1) == 1
    assert _call_compress(lib, cfg, FakeBatch([0, 4096, 4000])) == 1      # decreasing
    assert _call_compress(lib, cfg, FakeBatch([1, 4096])) == 1            # cu[0] != 0
    assert _call_compress(lib, cfg, b, q=None) == 1
    assert _call_compress(lib, cfg, b, k=_P + 8) == 1                     # misaligned
    assert _call_compress(lib, cfg, b, tok=1028) == 1                     # stride not % 8
    assert _call_compress(lib, cfg, b, head=-8) == 1
    assert _call_compress(lib, cfg, b, ws=None) == 3
    assert _call_compress(lib, cfg, b, ws=_P + 64) == 3                   # misaligned
    assert _call_compress(lib, cfg, b, ws_bytes=1024) == 3                # too small
    assert _call_compress(lib, cfg, b, cu_keep=None) == 1
    assert lib.ckv_compress_layer(None, 0, b.ref, _P, _P, _P, 0, 0, _P, _P, _P, _P, None, _P,
                                  1 << 30, None) == 1
    assert lib.ckv_compress_layer(cfg.ref, 0, None, _P, _P, _P, 0, 0, _P, _P, _P, _P, None, _P,
                                  1 << 30, None) == 1
    assert "workspace" in ckv.load().ckv_last_error_message().decode() or True


def _call_select(lib, cfg, batch, scores=_P, k=_P, v=_P, ws=_P, ws_bytes=1 << 30, cu_keep=_P):
    return lib.ckv_select_compact(cfg.ref, 0, batch.ref, scores, k, v, 0, 0, _P, cu_keep, _P, _P,
                                  None, ws, ws_bytes, None)


def test_select_compact_argument_errors(lib):
    """ckv_select_compact validates like ckv_compress_layer, plus its scores pointer (NULL or
    not 16-byte aligned); every check returns before a launch."""
    cfg, b = _cfg(), FakeBatch([0, 4096, 5000])
    assert _call_select(lib, cfg, b, scores=None) == 1
    assert b"scores" in lib.ckv_last_error_message()
    assert _call_select(lib, cfg, b, scores=_P + 4) == 1
    assert b"aligned" in lib.ckv_last_error_message()
    assert _call_select(lib, cfg, b, k=_P + 8) == 1
    assert _call_select(lib, cfg, b, ws=None) == 3
    assert _call_select(lib, cfg, b, ws_bytes=1024) == 3
    assert _call_select(lib, cfg, b, cu_keep=None) == 1
    assert _call_select(lib, cfg, FakeBatch([0, 4096, 4000])) == 1


def test_python_errors_carry_the_message(lib):
    cfg = _cfg(window=0)
    with pytest.raises(ckv.CkvError, match="window"):
        ckv.ckv_workspace_size(cfg, 0, FakeBatch([0, 10]))


@pytest.mark.skipif(__import__("torch").cuda.is_available(), reason="CPU-only behaviour")
def test_valid_call_without_a_gpu_reports_cuda_error(lib):
    rc = _call_compress(lib, _cfg(), FakeBatch([0, 4096]))
    assert rc == 4


def test_layer_scope_accepts_groups_without_heads(lib):
    """Per-layer selection: heads in one group only is a valid config (it gets past every host
    check, so on a machine without a GPU the call ends in CKV_ERR_CUDA)."""
    m = np.zeros((2, 32), np.uint8)
    m[:, :4] = 1
    assert _call_compress(lib, _cfg(scope=1, head_mask=m), FakeBatch([0, 4096])) in (0, 4)
    assert _call_compress(lib, _cfg(scope=0, head_mask=m), FakeBatch([0, 4096])) == 1


class _FakeT:
    """A stand-in device tensor for the binding: only its address matters on the host."""

    def __init__(self, addr):
        self.addr = addr

    def data_ptr(self):
        return self.addr


def _ios(n, **kw):
    out = []
    for i in range(n):
        d = dict(layer=i % 2, q_win=_FakeT(_P), k=_FakeT(_P), v=_FakeT(_P), scores=_FakeT(_P),
                 idx=_FakeT(_P), cu_keep_dev=_FakeT(_P), k_out=_FakeT(_P), v_out=_FakeT(_P))
        d.update(kw)
        out.append(ckv.LayerIO(**d))
    return out


def test_layers_workspace_grows_with_the_layers(lib):
    cfg, b = _cfg(), FakeBatch([0, 4096, 5000])
    one = ckv.ckv_workspace_size_layers(cfg, _ios(1), b)
    four = ckv.ckv_workspace_size_layers(cfg, _ios(4), b)
    assert one >= ckv.ckv_workspace_size(cfg, 0, b)
    # each extra layer adds its scores [n_sel, T] and its units' exchange
    assert four - one >= 3 * 8 * 5000 * 4


def test_layers_argument_errors(lib):
    cfg, b = _cfg(), FakeBatch([0, 4096, 5000])
    ios = _ios(3)
    arr = ckv._layer_ios(ios)
    assert lib.ckv_score_windows(cfg.ref, 0, arr, b.ref, _P, 1 << 30, None) == 1      # no layer
    assert lib.ckv_score_windows(cfg.ref, 3, None, b.ref, _P, 1 << 30, None) == 1     # io NULL
    assert lib.ckv_score_windows(cfg.ref, 3, arr, b.ref, _P, 1024, None) == 3         # too small
    assert lib.ckv_score_windows(cfg.ref, 3, arr, b.ref, _P + 64, 1 << 30, None) == 3  # misaligned
    bad = ckv._layer_ios(_ios(3, layer=5))
    assert lib.ckv_score_windows(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1      # layer range
    bad = ckv._layer_ios(_ios(2) + _ios(1, k=_FakeT(_P + 8)))
    assert lib.ckv_score_windows(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1      # misaligned k
    bad = ckv._layer_ios(_ios(3, scores=None))
    assert lib.ckv_score_windows(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1      # no scores
    bad = ckv._layer_ios(_ios(3, v=None))
    assert lib.ckv_compress_layers(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1    # no v
    bad = ckv._layer_ios(_ios(3, cu_keep_dev=None))
    assert lib.ckv_compress_layers(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1
    # the fused call needs room for every layer's scores; the scoring call does not
    need = ckv.ckv_workspace_size_layers(cfg, ios, b)
    assert lib.ckv_compress_layers(cfg.ref, 3, arr, b.ref, _P, need - 256, None) == 3
    # the given-lse form needs every layer's lse, aligned, with a head stride of at least S*w
    assert lib.ckv_compress_layers_lse(cfg.ref, 3, arr, b.ref, _P, 1 << 30, None) == 1   # no lse
    bad = ckv._layer_ios(_ios(3, lse=_FakeT(_P + 2)))
    assert lib.ckv_compress_layers_lse(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1   # misaligned
    bad = ckv._layer_ios(_ios(3, lse=_FakeT(_P), lse_head_stride=2 * 32 - 1))
    assert lib.ckv_compress_layers_lse(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1   # stride < S*w
    # the same checks in the scoring-only form
    assert lib.ckv_score_windows_lse(cfg.ref, 3, arr, b.ref, _P, 1 << 30, None) == 1     # no lse
    bad = ckv._layer_ios(_ios(3, lse=_FakeT(_P + 2)))
    assert lib.ckv_score_windows_lse(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1     # misaligned
    bad = ckv._layer_ios(_ios(3, lse=_FakeT(_P), lse_head_stride=2 * 32 - 1))
    assert lib.ckv_score_windows_lse(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1     # stride < S*w
    bad = ckv._layer_ios(_ios(2, lse=_FakeT(_P)) + _ios(1))
    assert lib.ckv_score_windows_lse(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1     # one missing
    bad = ckv._layer_ios(_ios(3, lse=_FakeT(_P), scores=None))
    assert lib.ckv_score_windows_lse(cfg.ref, 3, bad, b.ref, _P, 1 << 30, None) == 1     # no scores


@pytest.mark.skipif(__import__("torch").cuda.is_available(), reason="CPU-only behaviour")
def test_valid_layers_call_without_a_gpu_reports_cuda_error(lib):
    cfg, b = _cfg(), FakeBatch([0, 4096, 5000])
    arr = ckv._layer_ios(_ios(3))
    assert lib.ckv_score_windows(cfg.ref, 3, arr, b.ref, _P, 1 << 30, None) == 4
    assert lib.ckv_compress_layers(cfg.ref, 3, arr, b.ref, _P, 1 << 30, None) == 4
    arr = ckv._layer_ios(_ios(3, lse=_FakeT(_P)))
    assert lib.ckv_compress_layers_lse(cfg.ref, 3, arr, b.ref, _P, 1 << 30, None) == 4
    assert lib.ckv_score_windows_lse(cfg.ref, 3, arr, b.ref, _P, 1 << 30, None) == 4
