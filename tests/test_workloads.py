"""The seeded input generator: determinism, shapes and the stated recipes."""
import numpy as np

import workloads


def test_deterministic_and_shapes():
    wl = workloads.WORKLOADS["tiny"]
    a = workloads.reference_embeddings(wl)
    b = workloads.reference_embeddings(wl)
    assert a.shape == (256, 512) and a.dtype == np.float32
    np.testing.assert_array_equal(a, b)
    x, pos, src = workloads.target_prompt(wl, ref=a)
    assert x.shape == (256, 512) and (pos == np.arange(256)).all()
    assert (src == -1).sum() == 64  # 25% fresh rows


def test_bf16_rounding_of_inputs_is_nearest_even():
    v = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-39], dtype=np.float32)
    h = workloads.f32_to_bf16_bits(v)
    assert list(h[:4]) == [0x3F80, 0x3F80, 0x3F82, 0xC020]
    np.testing.assert_array_equal(workloads.bf16_bits_to_f32(h[:1]), [1.0])


def test_copied_rows_are_noisy_reference_rows():
    wl = workloads.WORKLOADS["llama8b-1k"].scaled(d=256)
    ref = workloads.reference_embeddings(wl)
    x, _, src = workloads.target_prompt(wl, ref=ref)
    rf = workloads.bf16_bits_to_f32(ref)
    xf = workloads.bf16_bits_to_f32(x)
    copied = src >= 0
    assert abs(copied.mean() - 0.70) < 1e-3
    resid = xf[copied] - rf[src[copied]]
    assert abs(resid.std() - wl.noise) < 0.01
    assert abs(xf[~copied].std() - 1.0) < 0.02


def test_window_recipe_moves_rows_locally():
    wl = workloads.WORKLOADS["llama8b-5k"].scaled(d=64)
    _, _, src = workloads.target_prompt(wl)
    copied = np.nonzero(src >= 0)[0]
    assert np.abs(src[copied] - copied).max() <= 2 * wl.window
    assert abs(len(copied) / wl.n_tgt - 0.5) < 1e-3


def test_subset_and_pool_recipes():
    wl = workloads.WORKLOADS["batched-64x2048"].scaled(d=64)
    _, _, s0 = workloads.target_prompt(wl, b=0)
    _, _, s1 = workloads.target_prompt(wl, b=1)
    c0 = s0[s0 >= 0]
    assert (np.diff(c0) > 0).all() and not np.array_equal(s0, s1)
    wp = workloads.WORKLOADS["pool-16x4096"].scaled(d=64)
    _, _, sp = workloads.target_prompt(wp)
    assert sp.max() < 65536 and len(np.unique(sp[sp >= 0] // 4096)) == 16
    assert (workloads.reference_positions(wp)[4096:4099] == [0, 1, 2]).all()


def test_kv_cache_segments():
    wl = workloads.WORKLOADS["tiny"]
    k, v = workloads.kv_cache(wl)
    assert k.shape == (1, 2, 4, 256, 64) and k.dtype == np.uint16
    k0, _ = workloads.kv_cache(wl, segment=0)
    np.testing.assert_array_equal(k0, k[0])


def test_retrieve_recipe_rewrites_one_member():
    wl = workloads.RETRIEVAL_WORKLOADS["retrieve-16x4096"].scaled(d=64)
    m = workloads.retrieval_member(wl)
    _, _, src = workloads.target_prompt(wl)
    copied = np.nonzero(src >= 0)[0]
    # copied rows come from the one member, in order, at their own position
    np.testing.assert_array_equal(src[copied], m * wl.seg_len + copied)
    assert abs(len(copied) / wl.n_tgt - wl.reuse) < 1e-3
    assert 0 <= m < wl.n_seg
