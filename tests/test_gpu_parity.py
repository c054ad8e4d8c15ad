"""Parity of the CUDA path (through the C ABI) with the fp64 oracle on seeded inputs.

Sizes span several key tiles, several chunks per (sequence, KV head), ragged tails, short and
empty sequences, every head-row padding width and both pooling orders; the five workloads are
run at full size on sampled layers (and sampled KV heads where the oracle would be slow).
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
    base = dict(name="fuzz", num_layers=2, num_q_heads=8, num_kv_heads=2, seqlens=(300,),
                window=32, heads_per_group=2, budget_mean=48, budget_uniform=True, pool_kernel=7,
                seed=11)
    base.update(kw)
    return cs.Workload(**base)


FUZZ = [
    dict(),
    dict(seqlens=(1, 5, 31, 32, 33, 127, 128, 129, 300, 0, 2000), budget_mean=40),
    dict(seqlens=(700, 129), budget_mean=32),                        # k = 0: the window only
    dict(window=8, pool_kernel=5, pool_type="avg", heads_per_group=4, seqlens=(1000,)),
    dict(window=8, pool_kernel=5, pool_type="avg", heads_per_group=4, seqlens=(1000, 77),
         head_order="sum_then_pool"),
    dict(window=17, heads_per_group=3, seqlens=(900, 450)),          # padded rows, 2 batches
    dict(window=64, heads_per_group=1, seqlens=(1500,), budget_mean=100),
    dict(window=64, heads_per_group=2, seqlens=(1500,), budget_mean=100),  # 2 batches of 1 head
    dict(window=1, heads_per_group=1, pool_kernel=1, seqlens=(513,), budget_mean=20),
    dict(window=16, heads_per_group=4, seqlens=(4096, 333), head_order="sum_then_pool"),
    dict(num_q_heads=28, num_kv_heads=4, heads_per_group=3, seqlens=(3000, 1200)),
    dict(num_q_heads=28, num_kv_heads=4, heads_per_group=7, window=8, seqlens=(2500,)),
    dict(num_q_heads=32, num_kv_heads=8, heads_per_group=2, seqlens=(8192,), budget_mean=256,
         outlier_channels=8),
    dict(seqlens=(5000,), plant="span", plant_count=32, plant_beta=4.0, plant_noise=True,
         budget_mean=64, pool_type="avg"),
    dict(seqlens=(20000,), budget_mean=600, heads_per_group=1, pool_kernel=9),
    # keys far above the rest, in later tiles of the work items: the column references move
    dict(seqlens=(3000, 1700), plant="tokens", plant_count=24, plant_beta=9.0, budget_mean=64),
    # one selection per layer from heads anywhere in the layer (Sec. 3.3 as stated)
    dict(scope="layer", heads_per_layer=3, seqlens=(1000, 77, 300), budget_mean=40),
    dict(scope="layer", heads_per_layer=4, num_q_heads=32, num_kv_heads=8, window=8,
         pool_kernel=5, pool_type="avg", seqlens=(4096, 333), budget_mean=128),
    dict(scope="layer", heads_per_layer=1, num_q_heads=28, num_kv_heads=4, seqlens=(20000, 3000),
         budget_mean=300, head_order="sum_then_pool"),
    dict(scope="layer", heads_per_layer=6, num_q_heads=32, num_kv_heads=8, window=64,
         seqlens=(1500, 9000), budget_mean=100),
    # pool kernels wider than the candidate range, L = w, L = w + 1, empty sequences
    dict(window=8, pool_kernel=9, seqlens=(12, 13, 9, 0, 17, 300, 8), budget_mean=10),
    dict(window=4, pool_kernel=63, heads_per_group=1, seqlens=(40, 70, 5, 0, 200), budget_mean=12,
         pool_type="avg"),
]


PATHS = [ckv.SCORE_RESIDENT, ckv.SCORE_RELOAD]


@pytest.mark.parametrize("path", PATHS, ids=["resident", "reload"])
@pytest.mark.parametrize("case", range(len(FUZZ)))
def test_fuzz_shapes(case, path):
    wl = _wl(**FUZZ[case])
    cfg = ckv.Config.from_workload(wl, score_path=path)
    for layer in range(wl.num_layers):
        li = wl.layer(layer)
        g = gu.run_gpu(wl, layer, li, cfg=cfg)
        o = gu.run_oracle(wl, layer, li)
        gu.check_layer(wl, layer, li, g, o)


def test_single_layer_workload_full():
    wl = cs.workload("single_layer_l2048")
    li = wl.layer(0)
    g = gu.run_gpu(wl, 0, li)
    o = gu.run_oracle(wl, 0, li)
    gu.check_layer(wl, 0, li, g, o)
    ck = o["cu_keep"]
    for gi in range(wl.num_kv_heads):  # the planted keys survive
        assert set(li.planted[0].tolist()) <= set(g["idx"][gi, ck[0]:ck[1]].tolist())


@pytest.mark.parametrize("name,layers,groups,path", [
    ("llama8b_l8192", (0, 13, 31), None, ckv.SCORE_AUTO),
    ("llama8b_l8192", (13,), None, ckv.SCORE_RELOAD),
    ("llama8b_l32768", (0, 5), None, ckv.SCORE_AUTO),
    ("needle_l131072", (7,), (0, 5), ckv.SCORE_AUTO),
    ("needle_l131072", (7,), (3,), ckv.SCORE_RELOAD),
    ("needle_l131072", (7,), (6,), ckv.SCORE_RESIDENT),
    ("llama8b_l8192", (5,), None, ckv.SCORE_RESIDENT),
    ("ragged_qwen7b", (0, 27), None, ckv.SCORE_AUTO),
    ("paper_llama8b_l8192", (0, 17, 31), None, ckv.SCORE_AUTO),
])
def test_full_size_workloads(name, layers, groups, path):
    wl = cs.workload(name)
    cfg = ckv.Config.from_workload(wl, score_path=path)
    for layer in layers:
        li = wl.layer(layer)
        g = gu.run_gpu(wl, layer, li, cfg=cfg, scores=groups is None)
        o = gu.run_oracle(wl, layer, li, groups=groups, want_kv=False)
        if groups is not None:
            g["scores"] = None
            g.pop("scores")
        gu.check_layer(wl, layer, li, g, o, groups=groups)
        if wl.plant == "tokens":  # the planted keys are kept by every KV head
            ck = o["cu_keep"]
            for gi in range(wl.num_kv_heads):
                assert set(li.planted[0].tolist()) <= set(g["idx"][gi, ck[0]:ck[1]].tolist())
        if wl.plant == "span":  # the needle span is kept by every KV head
            ck = o["cu_keep"]
            for gi in range(wl.num_kv_heads):
                assert set(li.planted[0].tolist()) <= set(g["idx"][gi, ck[0]:ck[1]].tolist())


@pytest.mark.parametrize("max_ctas", [9, 3])
def test_reload_kernel_over_many_rounds(max_ctas):
    """The reload kernel with its grid capped as the benchmark caps it: each CTA runs several
    rounds of items, so the double-buffered lse of the publisher warp is reused across rounds,
    and every unit has few enough items for that warp to combine them."""
    wl = cs.workload("llama8b_l8192")
    cfg = ckv.Config.from_workload(wl, score_path=ckv.SCORE_RELOAD, max_ctas=max_ctas)
    li = wl.layer(13)
    g = gu.run_gpu(wl, 13, li, cfg=cfg)
    o = gu.run_oracle(wl, 13, li, want_kv=False)
    gu.check_layer(wl, 13, li, g, o)


def test_unselected_heads_are_ignored():
    wl = _wl(seqlens=(3000, 400))
    li = wl.layer(0)
    a = gu.run_gpu(wl, 0, li)
    m = wl.head_mask()[0]
    li.q_win[:, :, m == 0, :] = 0x7FC0  # NaN in every unselected head
    b = gu.run_gpu(wl, 0, li)
    for key in ("scores", "pooled", "idx", "k_out", "v_out"):
        np.testing.assert_array_equal(np.nan_to_num(a[key]), np.nan_to_num(b[key]))


def test_deterministic():
    wl = _wl(seqlens=(6000, 300), num_q_heads=32, num_kv_heads=8)
    li = wl.layer(1)
    a = gu.run_gpu(wl, 1, li)
    b = gu.run_gpu(wl, 1, li)
    for key in ("scores", "pooled", "idx", "k_out", "v_out"):
        assert np.array_equal(a[key], b[key], equal_nan=True)


def test_standalone_entry_points_match_the_fused_call():
    wl = _wl(seqlens=(4000, 1000, 20), num_q_heads=32, num_kv_heads=8, pool_type="avg")
    layer = 0
    li = wl.layer(layer)
    cfg = ckv.Config.from_workload(wl)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k, v = gu.to_dev(li.q_win), gu.to_dev(li.k), gu.to_dev(li.v)
    ws = ckv.new_workspace(cfg, layer, batch)
    cu_keep, n_sel = ckv.ckv_keep_lengths(cfg, layer, batch)
    T, tk = batch.total_tokens, int(cu_keep[-1])
    guards = [gu.Guarded((n_sel, T), torch.float32), gu.Guarded((8, T), torch.float32),
              gu.Guarded((8, tk), torch.int32), gu.Guarded((4,), torch.int32),
              gu.Guarded((tk, 8, 128), torch.bfloat16), gu.Guarded((tk, 8, 128), torch.bfloat16)]
    scores, pooled, idx, cu_keep_dev, k_out, v_out = (g_.view for g_ in guards)
    ckv.ckv_score_window(cfg, layer, batch, q, k, scores, ws)
    ckv.ckv_pool(cfg, layer, batch, scores, pooled)
    ckv.ckv_select_topk(cfg, layer, batch, pooled, idx, cu_keep_dev, ws)
    ckv.ckv_gather_compact(cfg, batch, tk, k, v, idx, cu_keep_dev, k_out, v_out, ws)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    for g_ in guards:
        g_.check()
    fused = gu.run_gpu(wl, layer, li)
    np.testing.assert_array_equal(scores.cpu().numpy(), fused["scores"])
    np.testing.assert_array_equal(idx.cpu().numpy(), fused["idx"])
    np.testing.assert_array_equal(gu.to_host(k_out), fused["k_out"])
    np.testing.assert_array_equal(gu.to_host(v_out), fused["v_out"])
    # pooling: the GPU's pooled scores equal the oracle's pooling of the GPU's own scores
    sc = scores.cpu().numpy().astype(np.float64)
    pl = pooled.cpu().numpy()
    cu = wl.cu_seqlens()
    sel = np.nonzero(wl.head_mask()[layer])[0]
    for s in range(wl.num_seqs):
        t0, P = int(cu[s]), wl.seqlens[s] - wl.window
        if P <= 0:
            continue
        for gi in range(8):
            rows = [i for i, h in enumerate(sel) if h // 4 == gi]
            ref = sum(oracle.pool(sc[r, t0:t0 + P], wl.pool_kernel, 1) for r in rows)
            np.testing.assert_allclose(pl[gi, t0:t0 + P], ref, rtol=1e-5, atol=1e-30)


def test_split_score_and_select_match_the_fused_call():
    """ckv_score_window then ckv_select_compact (its own workspace, another stream) give the
    fused call's indices, pooled scores and gathered rows bit for bit."""
    wl = _wl(seqlens=(9000, 300, 20, 2500), num_q_heads=32, num_kv_heads=8)
    layer = 1
    li = wl.layer(layer)
    cfg = ckv.Config.from_workload(wl)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k, v = gu.to_dev(li.q_win), gu.to_dev(li.k), gu.to_dev(li.v)
    ws_score, ws_select = ckv.new_workspace(cfg, layer, batch), ckv.new_workspace(cfg, layer, batch)
    _, n_sel = ckv.ckv_keep_lengths(cfg, layer, batch)
    T = batch.total_tokens
    gsc = gu.Guarded((n_sel, T), torch.float32)
    gpl = gu.Guarded((cfg.num_vectors, T), torch.float32, float("nan"))
    *gouts, cu_keep = gu.guarded_outputs(cfg, layer, batch)
    scores, pooled = gsc.view, gpl.view
    idx, cu_keep_dev, k_out, v_out = (g_.view for g_ in gouts)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    ckv.ckv_score_window(cfg, layer, batch, q, k, scores, ws_score, stream=s1)
    ev = torch.cuda.Event()
    ev.record(s1)
    s2.wait_event(ev)
    ckv.ckv_select_compact(cfg, layer, batch, scores, k, v, idx, cu_keep_dev, k_out, v_out,
                           ws_select, pooled_out=pooled, stream=s2)
    torch.cuda.synchronize()
    assert ckv.ckv_read_device_status(ws_score) == (0, 0)
    assert ckv.ckv_read_device_status(ws_select) == (0, 0)
    for g_ in [gsc, gpl, *gouts]:
        g_.check()
    fused = gu.run_gpu(wl, layer, li)
    np.testing.assert_array_equal(idx.cpu().numpy(), fused["idx"])
    np.testing.assert_array_equal(cu_keep_dev.cpu().numpy(), fused["cu_keep_dev"])
    np.testing.assert_array_equal(gu.to_host(k_out), fused["k_out"])
    np.testing.assert_array_equal(gu.to_host(v_out), fused["v_out"])
    # sequences that fit the budget are not scored by the fused call: compare pooled elsewhere
    pl, fp = pooled.cpu().numpy(), fused["pooled"]
    cu = wl.cu_seqlens()
    for s_ in range(wl.num_seqs):
        if wl.seqlens[s_] > int(wl.budgets()[layer]):
            np.testing.assert_array_equal(pl[:, cu[s_]:cu[s_ + 1]], fp[:, cu[s_]:cu[s_ + 1]])
    with pytest.raises(ckv.CkvError, match="aligned"):
        ckv.ckv_select_compact(cfg, layer, batch, scores.view(-1)[1:], k, v, idx, cu_keep_dev,
                               k_out, v_out, ws_select)


def test_strided_kv_layout():
    """K and V interleaved in one [T, 2, H_kv, 128] buffer: strides select each half."""
    wl = _wl(seqlens=(2500, 700), num_q_heads=32, num_kv_heads=8)
    layer = 1
    li = wl.layer(layer)
    ref = gu.run_gpu(wl, layer, li)
    cfg = ref["cfg"]
    batch = ckv.Batch(wl.cu_seqlens())
    kv = torch.stack([gu.to_dev(li.k), gu.to_dev(li.v)], dim=1).contiguous()  # [T, 2, 8, 128]
    k_view, v_view = kv[:, 0], kv[:, 1]
    ws = ckv.new_workspace(cfg, layer, batch)
    *gouts, _ = gu.guarded_outputs(cfg, layer, batch)
    idx, cu_keep_dev, k_out, v_out = (g_.view for g_ in gouts)
    ckv.ckv_compress_layer(cfg, layer, batch, gu.to_dev(li.q_win), k_view, v_view, idx, cu_keep_dev,
                           k_out, v_out, ws, tok_stride=2 * 8 * 128, head_stride=128)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    for g_ in gouts:
        g_.check()
    np.testing.assert_array_equal(idx.cpu().numpy(), ref["idx"])
    np.testing.assert_array_equal(gu.to_host(k_out), ref["k_out"])
    np.testing.assert_array_equal(gu.to_host(v_out), ref["v_out"])


def test_device_lengths_that_disagree_are_reported():
    """cu_seqlens_dev splitting the same tokens differently from the host copy: the kernels
    stay in bounds and the status word says so."""
    wl = _wl(seqlens=(2000, 1000))
    li = wl.layer(0)
    cfg = ckv.Config.from_workload(wl)
    batch = ckv.Batch(wl.cu_seqlens(),
                      cu_seqlens_dev=torch.tensor([0, 1500, 3000], dtype=torch.int32, device="cuda"))
    ws = ckv.new_workspace(cfg, 0, batch)
    *gouts, _ = gu.guarded_outputs(cfg, 0, batch)
    idx, cu_keep_dev, k_out, v_out = (g_.view for g_ in gouts)
    ckv.ckv_compress_layer(cfg, 0, batch, gu.to_dev(li.q_win), gu.to_dev(li.k), gu.to_dev(li.v),
                           idx, cu_keep_dev, k_out, v_out, ws)
    code, _ = ckv.ckv_read_device_status(ws)
    assert code == 1
    for g_ in gouts:
        g_.check()
    assert ckv.ckv_read_device_status(ws) == (0, 0)  # the read reset it


@pytest.mark.parametrize("max_ctas,path", [(1, ckv.SCORE_AUTO), (5, ckv.SCORE_AUTO),
                                           (24, ckv.SCORE_RELOAD), (9, ckv.SCORE_RESIDENT),
                                           (24, ckv.SCORE_RESIDENT)])
def test_capped_grid_long_items_and_many_rounds(max_ctas, path):
    """A small CTA cap forces long work items (tiles re-loaded in pass 2, the only kernel that
    takes them) and several rounds; 9 CTAs is the fewest that fit 9000 tokens in TMEM."""
    wl = _wl(seqlens=(9000, 3000, 700), num_q_heads=32, num_kv_heads=8, budget_mean=300,
             outlier_channels=8)
    li = wl.layer(0)
    cfg = ckv.Config.from_workload(wl, max_ctas=max_ctas, score_path=path)
    g = gu.run_gpu(wl, 0, li, cfg=cfg)
    o = gu.run_oracle(wl, 0, li)
    gu.check_layer(wl, 0, li, g, o)


def test_resident_path_reports_what_does_not_fit():
    """9000 tokens are 71 key tiles: in TMEM (8 tiles per item at N = 64) they need 9 CTAs."""
    wl = _wl(seqlens=(9000,), num_q_heads=32, num_kv_heads=8, budget_mean=300)
    li = wl.layer(0)
    cfg = ckv.Config.from_workload(wl, max_ctas=8, score_path=ckv.SCORE_RESIDENT)
    with pytest.raises(ckv.CkvError, match="resident"):
        gu.run_gpu(wl, 0, li, cfg=cfg)
