"""Parity with the fp64 oracle on every layer, and every KV head, of every workload at full
size (Sec. 3.3; the layer budgets differ from layer to layer, so each layer selects a different
number of tokens), through both ckv_compress_layer (one layer per call) and
ckv_compress_layers (groups of layers per call).

Per layer: the pooled scores within the score tolerance, the indices exact (or, where the k-th
and (k+1)-th oracle scores are within the tolerance of each other, every token clearly above
the threshold kept and every token clearly below it dropped), the selection on the GPU's own
pooled scores exact, the window always kept, the gathered K/V rows bit-exact, planted keys kept
by every KV head, and canaries around every output buffer intact.
"""
import pytest
import torch

import ckv_synth as cs
import oracle
import paper_2508_02401_gb300 as ckv
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

WORKLOADS = ["single_layer_l2048", "llama8b_l8192", "llama8b_l32768", "needle_l131072",
             "ragged_qwen7b", "paper_llama8b_l8192"]
GROUP = 8  # layers per ckv_compress_layers call


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    ckv.load()
    oracle.build()


def _group_call(wl, cfg, layers, lis):
    """ckv_compress_layers over `layers`; per layer the outputs as gu.run_gpu returns them."""
    batch = ckv.Batch(wl.cu_seqlens())
    T = batch.total_tokens
    ios, outs = [], []
    for l, li in zip(layers, lis):
        gidx, gck, gk, gv, cu_keep = gu.guarded_outputs(cfg, l, batch)
        gpl = gu.Guarded((cfg.num_vectors, T), torch.float32, float("nan"))
        ios.append(ckv.LayerIO(layer=l, q_win=gu.to_dev(li.q_win), k=gu.to_dev(li.k),
                               v=gu.to_dev(li.v), idx=gidx.view, cu_keep_dev=gck.view,
                               k_out=gk.view, v_out=gv.view, pooled_out=gpl.view))
        outs.append((cu_keep, gidx, gck, gk, gv, gpl))
    ws = ckv.new_layers_workspace(cfg, ios, batch)
    ckv.ckv_compress_layers(cfg, ios, batch, ws)
    assert ckv.ckv_read_device_status(ws) == (0, 0)
    res = []
    for cu_keep, gidx, gck, gk, gv, gpl in outs:
        for g_ in (gidx, gck, gk, gv, gpl):
            g_.check()
        res.append(dict(cfg=cfg, cu_keep=cu_keep, pooled=gpl.view.cpu().numpy(),
                        idx=gidx.view.cpu().numpy(), cu_keep_dev=gck.view.cpu().numpy(),
                        k_out=gu.to_host(gk.view), v_out=gu.to_host(gv.view)))
    del ios, ws
    return res


def _planted_kept(wl, li, g, o, layer):
    if wl.plant == "none":
        return
    ck = o["cu_keep"]
    for s in range(wl.num_seqs):
        want = {int(x) for x in li.planted[s] if x >= 0}
        for gi in range(wl.num_kv_heads):
            assert want <= set(g["idx"][gi, ck[s]:ck[s + 1]].tolist()), (layer, s, gi)


@pytest.mark.parametrize("name", WORKLOADS)
def test_every_layer_of_the_workload(name):
    wl = cs.workload(name)
    cfg = ckv.Config.from_workload(wl)
    for l0 in range(0, wl.num_layers, GROUP):
        layers = list(range(l0, min(wl.num_layers, l0 + GROUP)))
        lis = [wl.layer(l) for l in layers]
        grouped = _group_call(wl, cfg, layers, lis)
        for layer, li, gg in zip(layers, lis, grouped):
            g = gu.run_gpu(wl, layer, li, cfg=cfg, scores=False)
            o = gu.run_oracle(wl, layer, li, want_kv=False)
            gu.check_layer(wl, layer, li, g, o)
            gu.check_layer(wl, layer, li, gg, o)
            _planted_kept(wl, li, g, o, layer)
            _planted_kept(wl, li, gg, o, layer)
        del lis, grouped
