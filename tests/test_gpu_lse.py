"""Parity of the single-pass scoring path (the window rows' lse given, as a prefill attention
kernel returns it) with the oracle, through the C ABI; and a decode-attention consumer check
over the compacted cache.

The lse fed to both sides is the oracle's own (fp64 rounded to fp32, natural log), laid out
[H_q, S*w] like a varlen prefill's per-head lse.  Tolerances as in gpu_util.
"""
import numpy as np
import pytest
import torch

import ckv_synth as cs
import oracle
import paper_2508_02401_gb300 as ckv
from tests import gpu_util as gu
from tests import independent as ind

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    ckv.load()
    oracle.build()


def _wl(**kw):
    base = dict(name="lse", num_layers=1, num_q_heads=8, num_kv_heads=2, seqlens=(300,),
                window=32, heads_per_group=2, budget_mean=48, budget_uniform=True, pool_kernel=7,
                seed=23)
    base.update(kw)
    return cs.Workload(**base)


def _oracle_lse(wl, li, pad=0):
    """[Hq, S*w + pad] float64: log sum_{j <= P+r} exp(scale q.k) per head and window row (NaN
    for rows before the sequence start), from the oracle's window attention."""
    cu = wl.cu_seqlens()
    S, w, Hq = wl.num_seqs, wl.window, wl.num_q_heads
    G = Hq // wl.num_kv_heads
    out = np.full((Hq, S * w + pad), np.nan)
    for s in range(S):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        for h in range(Hq):
            _, lse, _ = oracle.window_scores(li.q_win[s, :, h], li.k[t0:t1, h // G])
            out[h, s * w:(s + 1) * w] = lse
    return out


CASES = [
    dict(),
    dict(seqlens=(1, 5, 31, 32, 33, 127, 128, 129, 300, 0, 2000), budget_mean=40),
    dict(window=8, pool_kernel=5, pool_type="avg", heads_per_group=4, seqlens=(1000, 77)),
    dict(window=17, heads_per_group=3, seqlens=(900, 450)),
    dict(window=64, heads_per_group=2, seqlens=(1500,), budget_mean=100),
    dict(num_q_heads=32, num_kv_heads=8, heads_per_group=2, seqlens=(8192, 3000), budget_mean=256,
         outlier_channels=8),
    dict(seqlens=(3000, 1700), plant="tokens", plant_count=24, plant_beta=9.0, budget_mean=64),
    dict(scope="layer", heads_per_layer=4, num_q_heads=32, num_kv_heads=8, window=8,
         pool_kernel=5, pool_type="avg", seqlens=(4096, 333), budget_mean=128),
]


@pytest.mark.parametrize("case", range(len(CASES)))
@pytest.mark.parametrize("max_ctas", [0, 3])
def test_scores_and_layer_with_given_lse(case, max_ctas):
    wl = _wl(**CASES[case])
    li = wl.layer(0)
    pad = 5 if case % 2 else 0  # a padded head stride on every other case
    lse64 = _oracle_lse(wl, li, pad)
    o = oracle.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), wl.head_mask()[0],
                              int(wl.budgets()[0]), wl.window, wl.pool_kernel,
                              0 if wl.pool_type == "max" else 1,
                              0 if wl.head_order == "pool_then_sum" else 1,
                              scope=oracle.SCOPE_LAYER if wl.scope == "layer" else oracle.SCOPE_KV_HEAD,
                              lse=lse64)
    cfg = ckv.Config.from_workload(wl, max_ctas=max_ctas)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k, v = gu.to_dev(li.q_win), gu.to_dev(li.k), gu.to_dev(li.v)
    # NaN rows (before the sequence start) must never be read: poison them on the GPU side
    lse32 = torch.from_numpy(np.where(np.isnan(lse64), np.nan, lse64).astype(np.float32)).cuda()
    T = batch.total_tokens
    _, n_sel = ckv.ckv_keep_lengths(cfg, 0, batch)
    ws = ckv.new_workspace(cfg, 0, batch)
    gsc = gu.Guarded((n_sel, T), torch.float32, float("nan"))
    sc = gsc.view
    ckv.ckv_score_window_lse(cfg, 0, batch, q, k, lse32, sc, ws, lse_head_stride=lse64.shape[1])
    *gouts, cu_keep = gu.guarded_outputs(cfg, 0, batch)
    idx, cu_keep_dev, k_out, v_out = (g_.view for g_ in gouts)
    gpl = gu.Guarded((cfg.num_vectors, T), torch.float32, float("nan"))
    pooled = gpl.view
    ckv.ckv_compress_layer_lse(cfg, 0, batch, q, k, v, lse32, idx, cu_keep_dev, k_out, v_out, ws,
                               lse_head_stride=lse64.shape[1], pooled_out=pooled)
    code, detail = ckv.ckv_read_device_status(ws)
    assert code == 0, (code, detail)
    for g_ in [gsc, gpl, *gouts]:
        g_.check()
    g = dict(cfg=cfg, cu_keep=cu_keep, scores=sc.cpu().numpy(), pooled=pooled.cpu().numpy(),
             idx=idx.cpu().numpy(), cu_keep_dev=cu_keep_dev.cpu().numpy(),
             k_out=gu.to_host(k_out), v_out=gu.to_host(v_out))
    gu.check_layer(wl, 0, li, g, o)


def test_given_lse_agrees_with_the_computing_path():
    """The same layer through ckv_score_window (the kernel computes the lse) and through
    ckv_score_window_lse (the oracle's lse): both within the score tolerance of each other."""
    wl = _wl(num_q_heads=32, num_kv_heads=8, seqlens=(20000, 513), budget_mean=300)
    li = wl.layer(0)
    g1 = gu.run_gpu(wl, 0, li)
    cfg = ckv.Config.from_workload(wl)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k = gu.to_dev(li.q_win), gu.to_dev(li.k)
    lse32 = torch.from_numpy(_oracle_lse(wl, li).astype(np.float32)).cuda()
    _, n_sel = ckv.ckv_keep_lengths(cfg, 0, batch)
    gsc = gu.Guarded((n_sel, batch.total_tokens), torch.float32, float("nan"))
    sc = gsc.view
    ws = ckv.new_workspace(cfg, 0, batch)
    ckv.ckv_score_window_lse(cfg, 0, batch, q, k, lse32, sc, ws)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    gsc.check()
    gu.assert_close_rows(sc.cpu().numpy(), g1["scores"], rtol=2e-3)


def test_lse_argument_errors():
    wl = _wl()
    li = wl.layer(0)
    cfg = ckv.Config.from_workload(wl)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k = gu.to_dev(li.q_win), gu.to_dev(li.k)
    ws = ckv.new_workspace(cfg, 0, batch)
    sc = torch.empty((4, batch.total_tokens), dtype=torch.float32, device="cuda")
    lse = torch.zeros((8, 32), dtype=torch.float32, device="cuda")
    with pytest.raises(ckv.CkvError, match="lse_head_stride"):
        ckv.ckv_score_window_lse(cfg, 0, batch, q, k, lse, sc, ws, lse_head_stride=31)
    lib = ckv.load()
    rc = lib.ckv_score_window_lse(cfg.ref, 0, batch.ref, q.data_ptr(), k.data_ptr(), 0, 0,
                                  lse.data_ptr() + 2, 0, sc.data_ptr(), ws.data_ptr(), ws.numel(), None)
    assert rc == 1 and b"aligned" in lib.ckv_last_error_message()
    with pytest.raises(ckv.CkvError, match="NULL"):
        ckv.ckv_score_window_lse(cfg, 0, batch, q, k, None, sc, ws)


def _decode_attention(q, keys, vals):
    """softmax(q.K^T / sqrt(d)) V in float64 (one query, one KV head); also the probabilities."""
    s = keys @ q / np.sqrt(q.size)
    p = np.exp(s - s.max())
    p /= p.sum()
    return p @ vals, p


def test_decode_attention_over_the_compacted_cache():
    """A consumer of the compressed cache: decode attention of a fresh query over each
    sequence's kept rows.  Attending over the GPU's compacted rows equals attending over the
    input rows at the GPU's indices, and the planted keys (kept by every KV head) get at least
    the share of the attention they get over the whole sequence (removing other keys can only
    raise it)."""
    wl = cs.workload("single_layer_l2048").with_(seqlens=(2048, 900))
    li = wl.layer(0)
    g = gu.run_gpu(wl, 0, li, scores=False)
    cu, ck = wl.cu_seqlens(), g["cu_keep"]
    G = wl.num_q_heads // wl.num_kv_heads
    rng = np.random.default_rng(5)
    for s in range(wl.num_seqs):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        planted = set(int(x) for x in li.planted[s]) if s < len(li.planted) else set()
        for gi in range(wl.num_kv_heads):
            qd = ind.widen(li.q_win[s, :, gi * G]).mean(axis=0) + 0.01 * rng.standard_normal(wl.head_dim)
            rows = g["idx"][gi, ck[s]:ck[s + 1]]
            out_c, p_c = _decode_attention(qd, ind.widen(g["k_out"][ck[s]:ck[s + 1], gi]),
                                           ind.widen(g["v_out"][ck[s]:ck[s + 1], gi]))
            out_i, _ = _decode_attention(qd, ind.widen(li.k[t0 + rows, gi]), ind.widen(li.v[t0 + rows, gi]))
            np.testing.assert_allclose(out_c, out_i, rtol=1e-12, atol=1e-15)
            if planted and t1 - t0 > int(wl.budgets()[0]):
                _, p_f = _decode_attention(qd, ind.widen(li.k[t0:t1, gi]), ind.widen(li.v[t0:t1, gi]))
                kept = [i for i, r in enumerate(rows) if int(r) in planted]
                assert len(kept) == len(planted)
                assert p_c[kept].sum() >= p_f[sorted(planted)].sum() * (1 - 1e-12)


LAYERS_CASES = [
    dict(num_layers=3, num_q_heads=32, num_kv_heads=8, seqlens=(6000, 900), budget_mean=200,
         outlier_channels=8),
    dict(num_layers=2, seqlens=(5, 31, 300, 2500, 40), budget_mean=64),
    dict(num_layers=3, window=17, heads_per_group=3, num_q_heads=12, num_kv_heads=2,
         seqlens=(900, 450), budget_uniform=False),
    dict(num_layers=2, window=64, heads_per_group=2, seqlens=(1500, 700), budget_mean=100),
    dict(num_layers=3, scope="layer", heads_per_layer=4, num_q_heads=32, num_kv_heads=8, window=8,
         pool_kernel=5, pool_type="avg", seqlens=(4096, 333), budget_mean=128),
    # more layers than one launch takes (two scoring and two selection launches)
    dict(num_layers=34, num_q_heads=4, num_kv_heads=2, heads_per_group=1, seqlens=(600, 130),
         budget_mean=48),
    # more sequences than one launch's tables hold (the scoring in chunks of sequences)
    dict(num_layers=2, num_q_heads=2, num_kv_heads=1, heads_per_group=1, window=16,
         seqlens=tuple(100 + (i * 37) % 90 for i in range(600)), budget_mean=48),
]


# max_ctas: 0 = every SM; 5 and 1 = a capped grid, where each CTA takes many items in turn
# (the item ring wraps many times).
@pytest.mark.parametrize("max_ctas", [0, 5, 1])
@pytest.mark.parametrize("case", range(len(LAYERS_CASES)))
def test_layers_call_with_given_lse(case, max_ctas):
    """ckv_compress_layers_lse over several layers (every layer's single-pass scoring in one
    launch, then every layer's selection in one launch), and ckv_score_windows_lse (the scoring
    alone), against the oracle's layer with the same lse, layer by layer; canaries around every
    output.  Case 1: ragged lengths (some at most the
    budget, one shorter than the window) and a padded lse head stride; cases 2 and 3: 64-column
    MMAs (three heads of 17 rows, two of 64); case 4: one selection per layer; cases 5 and 6:
    more layers, or more sequences, than one launch takes."""
    wl = _wl(**LAYERS_CASES[case])
    pad = 3 * (case % 2)
    cfg = ckv.Config.from_workload(wl, max_ctas=max_ctas)
    batch = ckv.Batch(wl.cu_seqlens())
    T = batch.total_tokens
    ios, outs, refs = [], [], []
    for l in range(wl.num_layers):
        li = wl.layer(l)
        lse64 = _oracle_lse(wl, li, pad)
        refs.append((li, oracle.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), wl.head_mask()[l],
                                               int(wl.budgets()[l]), wl.window, wl.pool_kernel,
                                               0 if wl.pool_type == "max" else 1,
                                               0 if wl.head_order == "pool_then_sum" else 1,
                                               scope=oracle.SCOPE_LAYER if wl.scope == "layer"
                                               else oracle.SCOPE_KV_HEAD, lse=lse64)))
        lse32 = torch.from_numpy(lse64.astype(np.float32)).cuda()
        *gouts, cu_keep = gu.guarded_outputs(cfg, l, batch)
        gpl = gu.Guarded((cfg.num_vectors, T), torch.float32, float("nan"))
        _, n_sel = ckv.ckv_keep_lengths(cfg, l, batch)
        gsc = gu.Guarded((n_sel, T), torch.float32, float("nan"))
        ios.append(ckv.LayerIO(layer=l, q_win=gu.to_dev(li.q_win), k=gu.to_dev(li.k), v=gu.to_dev(li.v),
                               scores=gsc.view, idx=gouts[0].view, cu_keep_dev=gouts[1].view,
                               k_out=gouts[2].view, v_out=gouts[3].view, pooled_out=gpl.view, lse=lse32,
                               lse_head_stride=lse64.shape[1]))
        outs.append((gouts, gpl, gsc, cu_keep))
    ws = ckv.new_layers_workspace(cfg, ios, batch)
    ckv.ckv_compress_layers_lse(cfg, ios, batch, ws)
    code, detail = ckv.ckv_read_device_status(ws)
    assert code == 0, (code, detail)
    ckv.ckv_score_windows_lse(cfg, ios, batch, ws)  # the scoring alone, into io[i].scores
    code, detail = ckv.ckv_read_device_status(ws)
    assert code == 0, (code, detail)
    for l, ((gouts, gpl, gsc, cu_keep), (li, o)) in enumerate(zip(outs, refs)):
        for g_ in [gpl, gsc, *gouts]:
            g_.check()
        idx, cu_keep_dev, k_out, v_out = (g_.view for g_ in gouts)
        g = dict(cfg=cfg, cu_keep=cu_keep, scores=gsc.view.cpu().numpy(), pooled=gpl.view.cpu().numpy(),
                 idx=idx.cpu().numpy(), cu_keep_dev=cu_keep_dev.cpu().numpy(), k_out=gu.to_host(k_out),
                 v_out=gu.to_host(v_out))
        gu.check_layer(wl, l, li, g, o)
