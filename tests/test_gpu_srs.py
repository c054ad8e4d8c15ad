"""Parity of ckv_semantic_retrieval_scores (Sec. 3.2, Eq. 5) with the oracle, through the C ABI.

The decode steps' lse fed to the GPU is the oracle's own (fp64 rounded to fp32).  The score
tolerance of every other parity test applies: 1e-3 relative, plus 1e-12 of the largest head's
score.  Each head's score is a sum, over at most (answer span) x (decode steps) keys and steps,
of fp32 probabilities whose own relative error is about 1e-5 (the fp32 logit and exp2), and the
fp32 sums add at most another ~1e-4.
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


def _oracle_lse(wl, li):
    cu = wl.cu_seqlens()
    S, w, Hq = wl.num_seqs, wl.window, wl.num_q_heads
    G = Hq // wl.num_kv_heads
    out = np.full((Hq, S * w), np.nan)
    for s in range(S):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        for h in range(Hq):
            _, lse, _ = oracle.window_scores(li.q_win[s, :, h], li.k[t0:t1, h // G])
            out[h, s * w:(s + 1) * w] = lse
    return out


def _run(wl, flags, span, repeat=1, with_oracle=True):
    li = wl.layer(0)
    mask = np.ones((wl.num_layers, wl.num_q_heads), np.uint8)
    cfg = ckv.Config.from_workload(wl, head_mask=mask)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k = gu.to_dev(li.q_win), gu.to_dev(li.k)
    lse = torch.from_numpy(_oracle_lse(wl, li).astype(np.float32)).cuda()
    fl = torch.from_numpy(flags.astype(np.uint8)).cuda()
    sp = torch.from_numpy(span.astype(np.int32)).cuda()
    gsrs = gu.Guarded((wl.num_q_heads,), torch.float32, 0.0)
    srs = gsrs.view
    ws = ckv.new_workspace(cfg, 0, batch)
    for _ in range(repeat):
        ckv.ckv_semantic_retrieval_scores(cfg, 0, batch, q, k, lse, fl, sp, srs, ws)
    status = ckv.ckv_read_device_status(ws)
    gsrs.check()
    want = None
    if with_oracle:
        want = oracle.semantic_retrieval_scores(li.q_win, li.k, wl.cu_seqlens(), mask[0], wl.window,
                                                flags, span)
    return srs.cpu().numpy().astype(np.float64), want, status, li


CASES = [
    dict(seqlens=(300,), window=8),
    dict(seqlens=(1000, 77, 2500), window=16, num_q_heads=28, num_kv_heads=4),
    dict(seqlens=(4096,), window=32, num_q_heads=32, num_kv_heads=8, outlier_channels=8),
    dict(seqlens=(5, 40), window=8),  # a sequence shorter than the decode steps
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_srs_matches_the_oracle(case):
    base = dict(name="srs", num_layers=1, num_q_heads=8, num_kv_heads=2, heads_per_group=2,
                budget_mean=64, budget_uniform=True, seed=50 + case)
    base.update(CASES[case])
    wl = cs.Workload(**base)
    rng = np.random.default_rng(case)
    flags = (rng.random(wl.num_seqs * wl.window) < 0.6).astype(np.uint8)
    lens = np.diff(wl.cu_seqlens())
    span = np.array([[L // 3, L // 3 + max(1, L // 5)] for L in lens], np.int32)
    got, want, status, _ = _run(wl, flags, span, repeat=2)  # accumulates: twice the oracle's
    assert status == (0, 0)
    gu.assert_close_rows(got, 2 * want, what="srs")


def test_planted_span_heads_rank_first_on_the_gpu():
    wl = cs.Workload(name="srs", num_layers=1, num_q_heads=32, num_kv_heads=8, seqlens=(8192,),
                     window=16, heads_per_group=1, plant="span", plant_count=32, plant_beta=4.0,
                     budget_mean=256, budget_uniform=True, outlier_channels=8, seed=77)
    li = wl.layer(0)
    s0 = int(li.planted[0].min())
    got, want, status, _ = _run(wl, np.ones(wl.window, np.uint8), np.array([[s0, s0 + 32]], np.int32))
    assert status == (0, 0)
    gu.assert_close_rows(got, want, what="srs")
    mask = wl.head_mask()[0]
    for g in range(8):
        heads = range(4 * g, 4 * g + 4)
        top = max(heads, key=lambda h: got[h])
        assert mask[top]


def test_span_outside_the_sequence_is_reported():
    wl = cs.Workload(name="srs", num_layers=1, num_q_heads=8, num_kv_heads=2, seqlens=(300, 200),
                     window=8, heads_per_group=2, budget_mean=64, budget_uniform=True, seed=3)
    got, _, status, _ = _run(wl, np.ones(16, np.uint8), np.array([[10, 20], [150, 201]], np.int32),
                             with_oracle=False)
    assert status[0] == 3
