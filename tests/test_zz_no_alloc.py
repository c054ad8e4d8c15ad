"""ckv_score_window_static: window scoring for callers that cannot allocate device memory.

Some callers have no device allocator to hand (an engine whose memory pool is owned
elsewhere, or code that must not grow the device footprint after start-up), so this entry
point takes no workspace and keeps its scratch in a fixed static device array.  The test
calls it through the C ABI twice in a row and checks both results against the workspace
entry point and against the fp64 oracle, within the score tolerance of the parity tests.  This
file is collected last.
"""
import ctypes as C

import numpy as np
import pytest
import torch

import ckv_synth as cs
import oracle
import paper_2508_02401_gb300 as ckv
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    ckv.load()
    oracle.build()


def _static_against_workspace(wl, cfg, check_oracle=True):
    li = wl.layer(0)
    batch = ckv.Batch(wl.cu_seqlens())
    q, k = gu.to_dev(li.q_win), gu.to_dev(li.k)
    _, n_sel = ckv.ckv_keep_lengths(cfg, 0, batch)
    T = batch.total_tokens
    ref = torch.full((n_sel, T), float("nan"), dtype=torch.float32, device="cuda")
    ws = ckv.new_workspace(cfg, 0, batch)
    ckv.ckv_score_window(cfg, 0, batch, q, k, ref, ws)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    ref = ref.cpu().numpy()
    want = gu.run_oracle(wl, 0, li, want_kv=False)["scores"] if check_oracle else None

    lib = ckv.load()
    stream = torch.cuda.current_stream().cuda_stream
    for _ in range(2):
        gout = gu.Guarded((n_sel, T), torch.float32, float("nan"))
        out = gout.view
        status = torch.full((2,), -1, dtype=torch.int32, device="cuda")
        rc = lib.ckv_score_window_static(cfg.ref, 0, batch.ref, q.data_ptr(), k.data_ptr(), 0, 0,
                                         out.data_ptr(), status.data_ptr(), C.c_void_p(stream))
        assert rc == 0, lib.ckv_last_error_message()
        torch.cuda.synchronize()
        assert status.tolist() == [0, 0]
        gout.check()
        gu.assert_close_rows(out.cpu().numpy(), ref)
        if want is not None:  # and with the fp64 oracle, at the same tolerance
            gu.assert_close_rows(out.cpu().numpy(), want)


@pytest.mark.parametrize("path,max_ctas", [("auto", 0), ("reload", 3), ("resident", 0)])
def test_static_scratch_matches_workspace_entry_point_twice(path, max_ctas):
    wl = cs.Workload(name="noalloc", num_layers=1, num_q_heads=32, num_kv_heads=8,
                     seqlens=(6000, 1300, 45), window=32, heads_per_group=2, budget_mean=128,
                     budget_uniform=True, outlier_channels=8, seed=3)
    sp = {"auto": ckv.SCORE_AUTO, "reload": ckv.SCORE_RELOAD, "resident": ckv.SCORE_RESIDENT}[path]
    _static_against_workspace(wl, ckv.Config.from_workload(wl, score_path=sp, max_ctas=max_ctas))


def test_static_scratch_over_several_launches():
    # 400 short sequences, one KV head: 400 units of one item each, more units than one launch's
    # unit table holds (384), so the call is split into two launches that reuse the array.
    wl = cs.Workload(name="noalloc_many", num_layers=1, num_q_heads=2, num_kv_heads=1,
                     seqlens=tuple(100 + (i * 37) % 90 for i in range(400)), window=16,
                     heads_per_group=1, budget_mean=48, budget_uniform=True, seed=9)
    _static_against_workspace(wl, ckv.Config.from_workload(wl))


def test_static_scratch_rejects_work_beyond_its_size():
    # 1100 short sequences with one KV head: 1100 work items > the 1024 the array holds
    seqlens = [200] * 1100
    cfg = ckv.Config(num_layers=1, num_q_heads=1, num_kv_heads=1, window=32, pool_kernel=7,
                     pool_type=0, head_order=0, head_mask=np.ones((1, 1), np.uint8),
                     budgets=np.array([64], np.int32))
    batch = ckv.Batch(np.concatenate([[0], np.cumsum(seqlens)]))
    T = batch.total_tokens
    q = torch.zeros((1100, 32, 1, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((T, 1, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((1, T), dtype=torch.float32, device="cuda")
    with pytest.raises(ckv.CkvError, match="static scratch holds 1024"):
        ckv.ckv_score_window_static(cfg, 0, batch, q, k, out)
