"""Parity of the multi-layer calls (ckv_score_windows, ckv_compress_layers) with the fp64
oracle, layer by layer, through the C ABI: several layers' two passes in one persistent launch
(Sec. 3.3; every layer has its own head mask and budget).  Cases cover more layers than one
launch takes (two launches), more sequences than one launch takes (chunks of sequences),
layers whose head batches differ (one selection per layer from heads anywhere), both MMA
widths, short and empty sequences and a capped grid (long items, many rounds).  Every output
buffer sits between canaries.
"""
import numpy as np
import pytest
import torch

import ckv_synth as cs
import oracle
import paper_2508_02401_gb300 as ckv
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    ckv.load()
    oracle.build()


def _wl(**kw):
    base = dict(name="layers", num_layers=3, num_q_heads=8, num_kv_heads=2, seqlens=(3000, 700),
                window=32, heads_per_group=2, budget_mean=64, pool_kernel=7, seed=21)
    base.update(kw)
    return cs.Workload(**base)


CASES = [
    dict(num_q_heads=32, num_kv_heads=8, outlier_channels=8),
    dict(num_layers=2, seqlens=(1, 5, 31, 33, 300, 0, 2000), budget_mean=40, budget_uniform=True),
    dict(num_layers=4, scope="layer", heads_per_layer=3, seqlens=(1000, 77, 300), budget_mean=40),
    dict(num_layers=2, window=8, pool_kernel=5, pool_type="avg", heads_per_group=4, seqlens=(1000, 64)),
    dict(num_layers=2, window=64, heads_per_group=2, seqlens=(1500,), budget_mean=100,
         budget_uniform=True),
    dict(num_layers=34, num_q_heads=4, num_kv_heads=2, heads_per_group=1, seqlens=(600, 130),
         budget_mean=48),
    dict(num_layers=2, num_q_heads=2, num_kv_heads=1, heads_per_group=1, window=16,
         seqlens=tuple(100 + (i * 37) % 90 for i in range(600)), budget_mean=48),
    # three or four score rows per selection over several 8192-position chunks: the selection
    # stages them in one buffer
    dict(num_layers=2, num_q_heads=12, num_kv_heads=2, heads_per_group=3, seqlens=(20000, 9001),
         budget_mean=200),
    dict(num_layers=2, scope="layer", heads_per_layer=4, num_q_heads=32, num_kv_heads=8, window=8,
         pool_kernel=5, pool_type="avg", seqlens=(17000, 333), budget_mean=300),
]


def _run_layers(wl, cfg, lis, with_scores):
    batch = ckv.Batch(wl.cu_seqlens())
    T = batch.total_tokens
    ios, outs, guards = [], [], []
    for l, li in enumerate(lis):
        gidx, gck, gk, gv, cu_keep = gu.guarded_outputs(cfg, l, batch)
        gpl = gu.Guarded((cfg.num_vectors, T), torch.float32, float("nan"))
        _, n_sel = ckv.ckv_keep_lengths(cfg, l, batch)
        gsc = gu.Guarded((n_sel, T), torch.float32, float("nan"))
        ios.append(ckv.LayerIO(layer=l, q_win=gu.to_dev(li.q_win), k=gu.to_dev(li.k),
                               v=gu.to_dev(li.v), scores=gsc.view, idx=gidx.view,
                               cu_keep_dev=gck.view, k_out=gk.view, v_out=gv.view,
                               pooled_out=gpl.view))
        outs.append((cu_keep, gidx, gck, gk, gv, gpl, gsc))
        guards += [gidx, gck, gk, gv, gpl, gsc]
    ws = ckv.new_layers_workspace(cfg, ios, batch)
    ckv.ckv_compress_layers(cfg, ios, batch, ws)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    if with_scores:
        ckv.ckv_score_windows(cfg, ios, batch, ws)
        assert ckv.ckv_read_device_status(ws) == (0, 0)
    for g_ in guards:
        g_.check()
    res = []
    for cu_keep, gidx, gck, gk, gv, gpl, gsc in outs:
        g = dict(cfg=cfg, cu_keep=cu_keep, pooled=gpl.view.cpu().numpy(), idx=gidx.view.cpu().numpy(),
                 cu_keep_dev=gck.view.cpu().numpy(), k_out=gu.to_host(gk.view), v_out=gu.to_host(gv.view))
        if with_scores:
            g["scores"] = gsc.view.cpu().numpy()
        res.append(g)
    return res


# max_ctas: 0 = every SM, 5 = a capped grid (long items, many per CTA), 1 = one CTA (every unit
# one item, the whole launch in one CTA's two passes)
@pytest.mark.parametrize("max_ctas", [0, 5, 1])
@pytest.mark.parametrize("case", range(len(CASES)))
def test_layers_calls_match_the_oracle(case, max_ctas):
    wl = _wl(**CASES[case])
    cfg = ckv.Config.from_workload(wl, max_ctas=max_ctas)
    lis = [wl.layer(l) for l in range(wl.num_layers)]
    res = _run_layers(wl, cfg, lis, with_scores=True)
    for l, li in enumerate(lis):
        o = gu.run_oracle(wl, l, li, want_kv=False)
        gu.check_layer(wl, l, li, res[l], o)


def test_layers_call_equals_the_single_layer_calls():
    """The multi-layer call and ckv_compress_layer per layer select the same tokens."""
    wl = _wl(num_q_heads=32, num_kv_heads=8, seqlens=(9000, 2500, 40), budget_mean=200)
    cfg = ckv.Config.from_workload(wl, score_path=ckv.SCORE_RELOAD)
    lis = [wl.layer(l) for l in range(wl.num_layers)]
    res = _run_layers(wl, cfg, lis, with_scores=True)
    for l, li in enumerate(lis):
        one = gu.run_gpu(wl, l, li, cfg=cfg)
        gu.assert_close_rows(res[l]["scores"], one["scores"], rtol=2e-3)
        np.testing.assert_array_equal(res[l]["cu_keep_dev"], one["cu_keep_dev"])
        o = gu.run_oracle(wl, l, li, want_kv=False)
        gu.check_layer(wl, l, li, res[l], o)


def test_equal_scores_keep_the_lowest_positions():
    """Sequences whose keys are all zero give every candidate the same score (each window row
    spreads its mass evenly), so the multi-layer selection keeps the lowest positions.  The
    lengths take each of its tie paths: ties ranked by position in shared memory (168 equal
    keys), ties found by a scan of the scratch keys (268 and 1468), and more keys sharing the
    first digit than shared memory gathers (39968); the last sequence keeps random keys."""
    wl = _wl(num_layers=1, seqlens=(200, 300, 1500, 40000, 2500), budget_mean=64,
             budget_uniform=True)
    cfg = ckv.Config.from_workload(wl)
    li = wl.layer(0)
    cu = wl.cu_seqlens()
    for s in range(4):
        li.k[cu[s]:cu[s + 1]] = 0
    res = _run_layers(wl, cfg, [li], with_scores=True)
    o = gu.run_oracle(wl, 0, li, want_kv=False)
    gu.check_layer(wl, 0, li, res[0], o)
    ck = o["cu_keep"]
    for s in range(4):
        P = int(cu[s + 1] - cu[s]) - wl.window
        for g in range(wl.num_kv_heads):
            np.testing.assert_array_equal(res[0]["idx"][g, ck[s]:ck[s] + 32], np.arange(32))
            assert P > 32


def test_layers_call_with_interleaved_kv():
    """K and V interleaved in one [T, 2, H_kv, 128] buffer per layer, through the multi-layer
    call: the strides select each half, and the outputs equal those of the packed layout."""
    wl = _wl(num_q_heads=32, num_kv_heads=8, seqlens=(2500, 700, 9000))
    cfg = ckv.Config.from_workload(wl)
    lis = [wl.layer(l) for l in range(wl.num_layers)]
    packed = _run_layers(wl, cfg, lis, with_scores=False)
    batch = ckv.Batch(wl.cu_seqlens())
    ios, guards, keep = [], [], []
    for l, li in enumerate(lis):
        kv = torch.stack([gu.to_dev(li.k), gu.to_dev(li.v)], dim=1).contiguous()  # [T, 2, 8, 128]
        keep.append(kv)
        gidx, gck, gk, gv, _ = gu.guarded_outputs(cfg, l, batch)
        ios.append(ckv.LayerIO(layer=l, q_win=gu.to_dev(li.q_win), k=kv[:, 0], v=kv[:, 1],
                               idx=gidx.view, cu_keep_dev=gck.view, k_out=gk.view, v_out=gv.view,
                               tok_stride=2 * 8 * 128, head_stride=128))
        guards.append((gidx, gck, gk, gv))
    ws = ckv.new_layers_workspace(cfg, ios, batch)
    ckv.ckv_compress_layers(cfg, ios, batch, ws)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    for (gidx, gck, gk, gv), ref in zip(guards, packed):
        for g_ in (gidx, gck, gk, gv):
            g_.check()
        np.testing.assert_array_equal(gidx.view.cpu().numpy(), ref["idx"])
        np.testing.assert_array_equal(gu.to_host(gk.view), ref["k_out"])
        np.testing.assert_array_equal(gu.to_host(gv.view), ref["v_out"])
