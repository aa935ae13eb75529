"""Pins for the oracle's per-layer shared index set (Sec. 3.1: K is
H x N x D and the compressed cache is K[:, I, :], one I for all heads).

- A hand-worked example (tests/golden) that tells the Frobenius reading of
  a head block's cosine and norm from per-head averaging.
- Special cases: one head reduces to the per-head pass; identical heads give
  the per-head TaR and sqrt(H) times the VaN.
- Head-permutation invariance.
- Compaction of every head with its layer's indices.
Runs on CPU only.
"""
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _value(text):
    return {"1/sqrt(10)": 1 / math.sqrt(10), "-1/sqrt(2)": -1 / math.sqrt(2)}.get(text, None) \
        if "sqrt" in text else float(text)


def _load():
    meta, keys, vals, tar, van, sel = {}, [], [], {}, {}, []
    with open(os.path.join(GOLDEN, "shared_heads_worked_example.txt")) as fh:
        for line in fh:
            f = line.split("#", 1)[0].split()
            if not f:
                continue
            if f[0] in ("H", "D", "P", "N", "R"):
                meta[f[0]] = int(f[1])
            elif f[0] == "KEY":
                keys.append((int(f[1]), int(f[2]), float(f[3]), float(f[4])))
            elif f[0] == "VALUE":
                vals.append((int(f[1]), int(f[2]), float(f[3]), float(f[4])))
            elif f[0] == "TAR":
                tar[int(f[1])] = _value(f[2])
            elif f[0] == "VAN":
                van[int(f[1])] = _value(f[2])
            elif f[0] == "SELECT":
                sel.append((int(f[1]), float(f[2]), [int(x) for x in f[3:]]))
    H, N, D = meta["H"], meta["N"], meta["D"]
    K = np.zeros((H, N, D), np.float32)
    V = np.zeros((H, N, D), np.float32)
    for h, n, x, y in keys:
        K[h, n] = [x, y]
    for h, n, x, y in vals:
        V[h, n] = [x, y]
    return meta, K, V, tar, van, sel


def test_worked_example():
    meta, K, V, tar_x, van_x, sel = _load()
    H, N, p, r = meta["H"], meta["N"], meta["P"], meta["R"]
    tar, van = oracle.scores_shared(K, V, H, N, p, r)
    for n, x in tar_x.items():
        assert tar[0, n] == pytest.approx(x, abs=1e-15)
    for n, x in van_x.items():
        assert van[0, n] == x
    for budget, alpha, want in sel:
        kept = oracle.compress_shared(K, V, N, 1, p, r, budget, alpha, H)[0]
        assert kept[0].tolist() == want, (budget, alpha)


def test_one_head_is_the_per_head_pass():
    w = synth.CONFIGS["tiny"].scaled(n_layers=3, n_kv_heads=1)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    t1, v1 = oracle.scores(K, V, w.n_tokens, w.p, r)
    t2, v2 = oracle.scores_shared(K, V, 1, w.n_tokens, w.p, r)
    assert np.array_equal(t1, t2) and np.array_equal(v1, v2)
    a = oracle.compress(K, V, w.n_tokens, w.p, r, w.budget, w.tar_ratio)
    b = oracle.compress_shared(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget, w.tar_ratio, 1)
    for x, y in zip(a, b[:4]):
        assert np.array_equal(x, y)


def test_identical_heads():
    w = synth.CONFIGS["tiny"].scaled(n_layers=2, n_kv_heads=1)
    K1, V1 = synth.host_generate(w)
    K = np.repeat(K1, 4, axis=0)          # every layer's 4 heads are copies of one head
    V = np.repeat(V1, 4, axis=0)
    r = oracle.recent_frames(w.n_frames)
    t1, v1 = oracle.scores(K1, V1, w.n_tokens, w.p, r)
    t4, v4 = oracle.scores_shared(K, V, 4, w.n_tokens, w.p, r)
    np.testing.assert_allclose(t4, t1, rtol=0, atol=1e-14)
    np.testing.assert_allclose(v4, 2.0 * v1, rtol=1e-14, atol=0)   # sqrt(4) = 2


def test_head_order_does_not_matter():
    w = synth.CONFIGS["tiny"].scaled(n_layers=2, n_kv_heads=3)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    perm = np.array([2, 0, 1, 4, 5, 3])     # heads permuted within each layer
    a = oracle.scores_shared(K, V, 3, w.n_tokens, w.p, r)
    b = oracle.scores_shared(K[perm], V[perm], 3, w.n_tokens, w.p, r)
    for x, y in zip(a, b):
        np.testing.assert_allclose(x, y, rtol=1e-14, atol=1e-15)


def test_every_head_is_compacted_with_its_layers_indices():
    w = synth.CONFIGS["tiny"].scaled(n_layers=2, n_kv_heads=3)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    kept, kd, vd, pd, fd, _ = oracle.compress_shared(K, V, w.n_tokens, w.grid_h, w.grid_w, r,
                                                     w.budget, w.tar_ratio, 3)
    assert kept.shape == (2, w.budget)
    for s in range(6):
        idx = kept[s // 3]
        assert np.array_equal(kd[s, :w.budget], K[s, idx])
        assert np.array_equal(vd[s, :w.budget], V[s, idx])
        assert np.array_equal(pd[s, :w.budget], idx % w.p)
        assert np.array_equal(fd[s, :w.budget], idx // w.p)
    # the layer's TaR and VaN decide: the oracle's own selection on its scores
    tar, van = oracle.scores_shared(K, V, 3, w.n_tokens, w.p, r)
    assert np.array_equal(kept, oracle.select(tar, van, w.n_tokens, w.p, r, w.budget, w.tar_ratio))


def test_shared_pooled_at_pool_size_one_is_the_shared_pass():
    w = synth.CONFIGS["tiny"].scaled(n_layers=2, n_kv_heads=2)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    a = oracle.compress_shared(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget, w.tar_ratio, 2)
    b = oracle.compress_shared(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget, w.tar_ratio, 2,
                               tau=(0.0, 0.0, 0.0))
    for x, y in zip(a[:5], b[:5]):
        assert np.array_equal(x, y)
    # the layer's CV is over its shared VaN: VaN of every row of the layer
    all_v = oracle.van_all_shared(V, 2, w.n_tokens)
    t, v = oracle.scores_shared(K, V, 2, w.n_tokens, w.p, r)
    n_past = w.n_tokens - r * w.p
    assert np.array_equal(all_v[:, :n_past], v[:, :n_past])
