"""Parity with the fp64 oracle on every layer, and every KV head, of every workload at full
size, through ckv_compress_layer (Sec. 3.3; the layer budgets differ from layer to layer, so
each layer selects a different number of tokens).

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


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    ckv.load()
    oracle.build()


@pytest.mark.parametrize("name", WORKLOADS)
def test_every_layer_of_the_workload(name):
    wl = cs.workload(name)
    cfg = ckv.Config.from_workload(wl)
    for layer in range(wl.num_layers):
        li = wl.layer(layer)
        g = gu.run_gpu(wl, layer, li, cfg=cfg, scores=False)
        o = gu.run_oracle(wl, layer, li, want_kv=False)
        gu.check_layer(wl, layer, li, g, o)
        if wl.plant != "none":  # planted keys (a needle span) are kept by every KV head
            ck = o["cu_keep"]
            for s in range(wl.num_seqs):
                want = {int(x) for x in li.planted[s] if x >= 0}
                for gi in range(wl.num_kv_heads):
                    assert want <= set(g["idx"][gi, ck[s]:ck[s + 1]].tolist()), (layer, s, gi)
