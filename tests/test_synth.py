"""The seeded input generator: reproducibility, rounding and the workload recipe (CPU only)."""
import numpy as np
import pytest
import torch

import ckv_synth as cs


def test_bf16_rounding_matches_torch():
    x = np.concatenate([cs.normals(99, 100000) * 7, np.array([0.0, -0.0, 1.0, 1.00390625,
                                                              1.01171875, 3.4e38, 1e-40],
                                                             np.float32)]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(cs.bf16_bits(x), ref)
    np.testing.assert_array_equal(cs.bf16_to_f32(ref), torch.from_numpy(ref.view(np.int16))
                                  .view(torch.bfloat16).float().numpy())


def test_stream_is_counter_based():
    a = cs.uniform_u64(123, 0, 1000)
    b = cs.uniform_u64(123, 400, 600)
    np.testing.assert_array_equal(a[400:], b)
    n = cs.normals(5, 3001)
    np.testing.assert_array_equal(n[:1000], cs.normals(5, 1000))
    assert abs(n.mean()) < 0.08 and abs(n.std() - 1) < 0.05


def test_normal_statistics():
    z = cs.normals(2024, 1 << 21).astype(np.float64)
    assert abs(z.mean()) < 3e-3 and abs(z.var() - 1) < 5e-3
    assert abs((z ** 3).mean()) < 1e-2 and abs((z ** 4).mean() - 3) < 3e-2


def test_layers_are_independent_and_reproducible():
    wl = cs.workload("single_layer_l2048").with_(num_layers=3, budget_uniform=True)
    a = wl.layer(2)
    _ = wl.layer(0)
    b = wl.layer(2)
    for f in ("q_win", "k", "v", "planted"):
        np.testing.assert_array_equal(getattr(a, f), getattr(b, f))
    assert not np.array_equal(wl.layer(1).k, a.k)


@pytest.mark.parametrize("name", cs.WORKLOAD_ORDER)
def test_workload_recipe(name):
    wl = cs.workload(name)
    m = wl.head_mask()
    assert m.shape == (wl.num_layers, wl.num_q_heads)
    if wl.heads_per_layer > 0:  # that many heads per layer, anywhere in the layer
        assert np.all(m.sum(-1) == wl.heads_per_layer)
        assert len({tuple(np.nonzero(r)[0]) for r in m}) > 1  # layers differ
    else:
        per_group = m.reshape(wl.num_layers, wl.num_kv_heads, wl.group_size).sum(-1)
        assert np.all(per_group == wl.heads_per_group)
    b = wl.budgets()
    assert b.sum() == wl.num_layers * wl.budget_mean
    assert b.min() >= max(wl.budget_min, wl.window) and b.max() <= 3 * wl.budget_mean
    if not wl.budget_uniform and wl.num_layers > 1:
        assert len(set(b.tolist())) > 1
    cu = wl.cu_seqlens()
    assert cu[0] == 0 and np.all(np.diff(cu) >= 0) and cu[-1] == wl.total_tokens


def test_planted_keys_follow_the_recipe():
    wl = cs.workload("single_layer_l2048")
    li = wl.layer(0)
    pos = li.planted[0]
    assert len(pos) == 4 and np.all(pos < 2048 - 32)
    m = wl.head_mask()[0]
    q = cs.bf16_to_f32(li.q_win).astype(np.float64)
    for g in range(wl.num_kv_heads):
        heads = np.nonzero(m[g * 4:(g + 1) * 4])[0] + g * 4
        u = q[0][:, heads, :].reshape(-1, 128).mean(0)
        u /= np.linalg.norm(u)
        k = cs.bf16_to_f32(li.k[pos, g, :]).astype(np.float64)
        np.testing.assert_allclose(k, np.tile(6.0 * np.sqrt(128) * u, (4, 1)), rtol=1e-2, atol=0.02)


def test_outlier_channels_present():
    wl = cs.workload("llama8b_l8192").with_(seqlens=(4096,))
    k = cs.bf16_to_f32(wl.layer(0).k)
    std = k.std(axis=0)  # [Hkv, d]
    for g in range(wl.num_kv_heads):
        big = np.sort(std[g])[-8:]
        assert np.all(big > 8) and np.sort(std[g])[-9] < 1.2


def test_span_plant_is_contiguous():
    wl = cs.workload("needle_l131072").with_(seqlens=(4096,), num_layers=2)
    li = wl.layer(1)
    span = li.planted[0]
    assert np.all(np.diff(span) == 1) and len(span) == 64 and span[-1] < 4096 - 32


def test_bulk_draws_equal_the_numpy_stream():
    """The C library's draws are the numpy definition of the stream, bit for bit."""
    for key, start, n in ((7, 0, 1000), (2**63 + 12345, 999, 4097), (0, 10**9, 64)):
        np.testing.assert_array_equal(cs.uniform_u64_fast(key, start, n), cs.uniform_u64(key, start, n))


def test_bf16_normals_are_the_rounded_float32_normals():
    scale = np.array([1.0, 10.0, 0.5], np.float32)
    n = cs.normals(77, 3001)
    np.testing.assert_array_equal(cs.normals_bf16(77, 3001), cs.bf16_bits(n))
    np.testing.assert_array_equal(cs.normals_bf16(77, 3001, scale),
                                  cs.bf16_bits(n * np.resize(scale, 3001)))
