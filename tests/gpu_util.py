"""Helpers for the GPU parity tests: run the CUDA path through the C ABI and compare with the
oracle under the tolerances of the parity contract.

Tolerances (the GPU accumulates in fp32, the oracle in fp64):
  * scores, pooled:  |gpu - oracle| <= 1e-3 * |oracle| + 1e-12 * max(oracle of that row)
    (the floor absorbs fp32 underflow of probabilities that are negligible in the row);
  * pooling of the GPU's own scores: 1e-5 relative (a handful of fp32 roundings);
  * selection on the GPU's own pooled scores: bit-exact (same fp32 values, same decision);
  * selection against the oracle's scores: exact unless the k-th and (k+1)-th oracle scores
    are within 1e-3 of each other, otherwise every token clearly above / below the threshold
    band must be in / out;
  * gathered K/V: bit-exact against the input rows at the GPU's indices.

Every output buffer of `run_gpu` sits between canary bytes that are checked after the calls:
a kernel that writes past an output's end (or before its start) fails the test.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2508_02401_gb300 as ckv

SCORE_RTOL = 1e-3
SCORE_FLOOR = 1e-12


def to_dev(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def to_host(t: torch.Tensor) -> np.ndarray:
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


GUARD_BYTES = 4096          # canary bytes before and after every output buffer
GUARD_BYTE = 0xA5


class Guarded:
    """A device buffer with canary bytes on both sides: `view` is what the library writes;
    `check()` asserts that nothing was written outside it (compute-sanitizer stands in)."""

    def __init__(self, shape, dtype, fill=None):
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        self.raw = torch.full((GUARD_BYTES + n + GUARD_BYTES,), GUARD_BYTE, dtype=torch.uint8,
                              device="cuda")
        self.view = self.raw[GUARD_BYTES:GUARD_BYTES + n].view(dtype).view(shape)
        if fill is not None:
            self.view.fill_(fill)
        self.what = f"{tuple(shape)} {dtype}"

    def check(self):
        head = self.raw[:GUARD_BYTES].cpu().numpy()
        tail = self.raw[-GUARD_BYTES:].cpu().numpy()
        assert np.all(head == GUARD_BYTE) and np.all(tail == GUARD_BYTE), \
            f"a kernel wrote outside the output buffer {self.what}"


def guarded_outputs(cfg, layer, batch):
    """(idx, cu_keep_dev, k_out, v_out) as canary-guarded buffers, and the host cu_keep."""
    cu_keep, _ = ckv.ckv_keep_lengths(cfg, layer, batch)
    tk = int(cu_keep[-1])
    H = cfg.num_kv_heads
    return (Guarded((H, tk), torch.int32, -7), Guarded((batch.num_seqs + 1,), torch.int32, -7),
            Guarded((tk, H, 128), torch.bfloat16), Guarded((tk, H, 128), torch.bfloat16), cu_keep)


def run_gpu(wl, layer, li, cfg=None, scores=True, stream=None, check_status=True):
    """compress_layer (+ score_window when asked) for one layer; numpy outputs.  Every output
    buffer carries canaries on both sides, checked after the calls."""
    cfg = cfg or ckv.Config.from_workload(wl)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k, v = to_dev(li.q_win), to_dev(li.k), to_dev(li.v)
    ws = ckv.new_workspace(cfg, layer, batch)
    gidx, gck, gk, gv, cu_keep = guarded_outputs(cfg, layer, batch)
    T = batch.total_tokens
    gpooled = Guarded((cfg.num_vectors, T), torch.float32, float("nan"))
    ckv.ckv_compress_layer(cfg, layer, batch, q, k, v, gidx.view, gck.view, gk.view, gv.view, ws,
                           pooled_out=gpooled.view, stream=stream)
    guards = [gidx, gck, gk, gv, gpooled]
    out = dict(cfg=cfg, cu_keep=cu_keep)
    if scores:
        _, n_sel = ckv.ckv_keep_lengths(cfg, layer, batch)
        gsc = Guarded((n_sel, T), torch.float32, float("nan"))
        ckv.ckv_score_window(cfg, layer, batch, q, k, gsc.view, ws, stream=stream)
        guards.append(gsc)
        out["scores"] = gsc.view.cpu().numpy()
    code, detail = ckv.ckv_read_device_status(ws, stream=stream)
    if check_status:
        assert code == 0, f"device status {code} ({detail})"
    for g in guards:
        g.check()
    out.update(status=(code, detail), pooled=gpooled.view.cpu().numpy(), idx=gidx.view.cpu().numpy(),
               cu_keep_dev=gck.view.cpu().numpy(), k_out=to_host(gk.view), v_out=to_host(gv.view))
    return out


def run_oracle(wl, layer, li, mask=None, groups=None, want_kv=True):
    m = wl.head_mask()[layer] if mask is None else mask
    return oracle.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), m,
                                 int(wl.budgets()[layer]), wl.window, wl.pool_kernel,
                                 0 if wl.pool_type == "max" else 1,
                                 0 if wl.head_order == "pool_then_sum" else 1,
                                 want_kv=want_kv, groups=groups,
                                 scope=oracle.SCOPE_LAYER if wl.scope == "layer" else oracle.SCOPE_KV_HEAD)


def assert_close_rows(gpu, orc, rtol=SCORE_RTOL, floor=SCORE_FLOOR, what="scores"):
    gpu = np.asarray(gpu, np.float64)
    orc = np.asarray(orc, np.float64)
    assert gpu.shape == orc.shape
    if orc.size == 0:
        return
    tol = rtol * np.abs(orc) + floor * np.max(np.abs(orc))
    bad = ~(np.abs(gpu - orc) <= tol)
    if bad.any():
        i = np.argmax(np.where(bad, np.abs(gpu - orc) / (np.abs(orc) + 1e-300), 0))
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside tolerance; worst at {i}: "
                             f"gpu={gpu.flat[i]!r} oracle={orc.flat[i]!r}")


def check_layer(wl, layer, li, g, o, groups=None, exact_select=True):
    """All parity checks of one layer: g = run_gpu output, o = run_oracle output."""
    cu = wl.cu_seqlens()
    B = int(wl.budgets()[layer])
    w = wl.window
    np.testing.assert_array_equal(g["cu_keep"], o["cu_keep"])
    np.testing.assert_array_equal(g["cu_keep_dev"], o["cu_keep"])
    ck = o["cu_keep"]
    groups = range(wl.num_kv_heads) if groups is None else groups
    sel_rows = np.nonzero(wl.head_mask()[layer])[0]
    G = wl.group_size
    layer_scope = wl.scope == "layer"
    if layer_scope:  # one selection per sequence, the same positions for every KV head
        for gi in groups:
            np.testing.assert_array_equal(g["idx"][gi], g["idx"][0])
    for s in range(wl.num_seqs):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        L = t1 - t0
        P = L - w
        for gi in groups:  # scores of the group's selected heads, every position
            if "scores" in g and L > 0:
                rows = [i for i, h in enumerate(sel_rows) if h // G == gi]
                assert_close_rows(g["scores"][rows, t0:t1], o["scores"][rows, t0:t1])
        for gi in ([0] if layer_scope else groups):  # the selections
            ix = g["idx"][gi, ck[s]:ck[s + 1]]
            if L <= B:
                np.testing.assert_array_equal(ix, np.arange(L))
                continue
            k = B - w
            assert_close_rows(g["pooled"][gi, t0:t0 + P], o["pooled"][gi, t0:t0 + P], what="pooled")
            np.testing.assert_array_equal(ix[k:], np.arange(P, L))
            cand = ix[:k]
            assert np.all(np.diff(cand) > 0) and (k == 0 or (cand[0] >= 0 and cand[-1] < P))
            if exact_select:
                # the selection, decided on the GPU's own fp32 pooled scores, is exact
                np.testing.assert_array_equal(
                    cand, oracle.topk(g["pooled"][gi, t0:t0 + P].astype(np.float64), k))
            # against the oracle's fp64 scores: exact unless the k-th / (k+1)-th are too close
            c = o["pooled"][gi, t0:t0 + P]
            if k == 0:
                continue
            order = np.lexsort((np.arange(P), -c))
            ck_, floor = c[order[k - 1]], SCORE_FLOOR * c.max()
            band = SCORE_RTOL * ck_ + floor
            cs = set(cand.tolist())
            assert set(np.nonzero(c > ck_ + band)[0].tolist()) <= cs
            assert not (set(np.nonzero(c < ck_ - band)[0].tolist()) & cs)
            if k < P and c[order[k - 1]] - c[order[k]] >= band:
                assert cs == set(order[:k].tolist())
    # gathered rows are the input rows at the GPU's indices, bit for bit
    for s in range(wl.num_seqs):
        for gi in groups:
            rows = cu[s] + g["idx"][gi, ck[s]:ck[s + 1]]
            np.testing.assert_array_equal(g["k_out"][ck[s]:ck[s + 1], gi], li.k[rows, gi])
            np.testing.assert_array_equal(g["v_out"][ck[s]:ck[s + 1], gi], li.v[rows, gi])
