"""The seeded input generator follows its stated recipe (CPU)."""
import numpy as np

import synth


def test_philox_known_answers():
    """Philox4x32-10 known-answer vectors published with Random123."""
    r = synth.philox4x32_10((0, 0, 0, 0), (0, 0))
    assert [int(x) for x in r] == [0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8]
    r = synth.philox4x32_10((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2)
    assert [int(x) for x in r] == [0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD]
    r = synth.philox4x32_10((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344),
                            (0xA4093822, 0x299F31D0))
    assert [int(x) for x in r] == [0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1]


def test_patch_kinds():
    for name in ("tiny", "llava", "qwen"):
        w = synth.CONFIGS[name]
        rho = synth.patch_rho(w)
        assert (rho == np.float32(w.rho_static)).sum() == int(np.floor(w.static_frac * w.p))
        assert np.array_equal(rho, synth.patch_rho(w))          # seeded
    w = synth.CONFIGS["llava"]
    assert not np.array_equal(synth.patch_rho(w, 0), synth.patch_rho(w, 1))


def test_key_and_value_statistics():
    w = synth.CONFIGS["llava"].scaled(n_layers=1, n_kv_heads=2, n_frames=24, head_dim=64)
    K, V = synth.host_generate(w)
    K = synth.bf16_bits_to_f32(K).astype(np.float64).reshape(2, w.n_frames, w.p, w.head_dim)
    V = synth.bf16_bits_to_f32(V).astype(np.float64)
    rho = synth.patch_rho(w)
    for kind in (w.rho_static, w.rho_dynamic):
        q = np.nonzero(rho == np.float32(kind))[0]
        a, b = K[:, :-1, q].ravel(), K[:, 1:, q].ravel()
        assert abs(np.corrcoef(a, b)[0, 1] - kind) < 0.05
    dyn = np.nonzero(rho == np.float32(w.rho_dynamic))[0]
    var = K[:, :, dyn].var()
    assert abs(var - 1 / (1 - w.rho_dynamic ** 2)) < 0.1          # stationary variance
    lognorm = np.log(np.linalg.norm(V, axis=-1)).ravel()
    assert abs(lognorm.mean()) < 0.03 and abs(lognorm.std() - w.value_sigma) < 0.03


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-3], np.float32)
    b = synth.to_bf16_bits(x)
    back = synth.bf16_bits_to_f32(b)
    assert b[1] == 0x3F80 and b[2] == 0x3F82       # ties to even
    assert np.all(np.abs(back - x) <= np.abs(x) * 2 ** -8)


def test_layer_varying_values():
    """Per-layer value spread and spatial clustering (the pooled workload):
    the log-norm spread of layer l is sigma_l; the smooth field makes
    neighbouring patches of a frame correlated in early layers only."""
    w = synth.CONFIGS["llava_pool"].scaled(n_layers=4, n_kv_heads=2, n_frames=16, head_dim=32,
                                           budget=1000)
    sig, beta = synth.value_params(w)
    assert np.allclose(sig, [0.25, 0.5, 0.75, 1.0]) and np.allclose(beta, [0.9, 0.6, 0.3, 0.0])
    _, V = synth.host_generate(w)
    V = synth.bf16_bits_to_f32(V).astype(np.float64)
    ln = np.log(np.linalg.norm(V, axis=-1)).reshape(w.n_layers, w.n_kv_heads, w.n_frames,
                                                    w.grid_h, w.grid_w)
    corr = []
    for layer in range(w.n_layers):
        x = ln[layer]
        assert abs(x.std() - sig[layer]) < 0.08 * sig[layer] + 0.02
        a, b = x[..., :, :-1].ravel(), x[..., :, 1:].ravel()     # horizontal neighbours
        corr.append(np.corrcoef(a, b)[0, 1])
    assert corr[0] > 0.5 and abs(corr[-1]) < 0.1 and corr[0] > corr[1] > corr[2]
    # defaults leave every layer at value_sigma with no field
    assert synth.value_params(synth.CONFIGS["llava"]) is None


def test_host_generation_of_a_slab_range_is_a_slice_of_the_whole():
    """Slabs generated from an offset (the reference arm generates ranges in
    parallel) equal the same slabs of one whole generation."""
    w = synth.Workload("rng", 3, 2, 64, "bf16", 3, 4, 5, 24, 0.5, seed=9)
    K, V = synth.host_generate(w)
    K2, V2 = synth.host_generate(w, slabs=3, slab0=2)
    assert np.array_equal(K[2:5], K2) and np.array_equal(V[2:5], V2)
    wp = synth.CONFIGS["llava_pool"].scaled(n_layers=3, n_frames=3, grid_h=3, grid_w=3, budget=18)
    Kp, Vp = synth.host_generate(wp)
    Kq, Vq = synth.host_generate(wp, slabs=5, slab0=6)  # per-layer value parameters follow the slab
    assert np.array_equal(Kp[6:11], Kq) and np.array_equal(Vp[6:11], Vq)
