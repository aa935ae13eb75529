"""Pins for the oracle's layer-adaptive VaN pooling (Sec. 3.2 "Layer-wise
Adaptive Pooling"; Algorithm 2: CV = sigma/mu per layer, pool size g(CV),
AveragePool2d over each frame's VaN map).

Each test ties the oracle to something other than itself:
- the case table of g;
- CV closed forms that tell population from sample deviation and layer from head;
- a hand-worked compacted-cache example (tests/golden);
- torch's avg_pool2d on whole frames, a library routine;
- the k = 1 identity;
- exact power-of-two scaling;
- frame independence.
Runs on CPU only.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
INF = float("inf")
FORCE = {7: (INF, INF, INF), 5: (0.0, INF, INF), 3: (0.0, 0.0, INF), 1: (0.0, 0.0, 0.0)}


def test_pool_size_cases():
    tau = (0.2, 0.5, 0.8)
    assert oracle.pool_size(0.0, tau) == 7
    assert oracle.pool_size(0.19999, tau) == 7
    assert oracle.pool_size(0.2, tau) == 5          # tau_1 <= CV < tau_2
    assert oracle.pool_size(0.49999, tau) == 5
    assert oracle.pool_size(0.5, tau) == 3
    assert oracle.pool_size(0.8, tau) == 1          # CV >= tau_3
    assert oracle.pool_size(5.0, tau) == 1
    assert oracle.pool_size(float("nan"), tau) == 1


def test_cv_population_std_over_the_whole_layer():
    # One layer of two heads: head 0 all 1, head 1 all 3. Layer mu = 2,
    # population sigma = 1 -> CV = 0.5 exactly; each head alone has CV 0.
    N = 8
    van = np.stack([np.ones(N), np.full(N, 3.0)])
    _, ks, cv = oracle.van_pool(van, 2, 2, 4, (0.45, 0.55, 0.9))
    assert cv[0] == 0.5 and ks[0] == 5
    # At the boundary CV == tau_1 the pool size is 5, not 7.
    assert oracle.van_pool(van, 2, 2, 4, (0.5, 0.9, 1.0))[1][0] == 5
    # 4 values {1,1,3,3}: population sigma 1 (CV 0.5), sample sigma sqrt(4/3)
    # (CV 0.577): tau_1 = 0.55 separates them.
    van4 = np.array([[1.0, 3.0, 1.0, 3.0]])
    _, ks, cv = oracle.van_pool(van4, 1, 1, 2, (0.55, 0.9, 1.0))
    assert cv[0] == 0.5 and ks[0] == 7
    # Two layers get their own CV.
    van2 = np.concatenate([van, np.ones((2, N))])
    _, ks, cv = oracle.van_pool(van2, 2, 2, 4, (0.45, 0.55, 0.9))
    assert list(ks) == [5, 7] and cv[1] == 0.0


def _load_worked_example():
    rows, pools = [], []
    with open(os.path.join(GOLDEN, "van_pool_worked_example.txt")) as fh:
        for line in fh:
            f = line.split("#", 1)[0].split()
            if not f:
                continue
            if f[0] == "GRID":
                gh, gw = int(f[1]), int(f[2])
            elif f[0] == "ROW":
                rows.append((int(f[1]), int(f[2]), float(f[3])))
            elif f[0] == "POOL":
                pools.append((int(f[1]), int(f[2]), float(Fraction(f[3]))))
    return gh, gw, rows, pools


def test_worked_example_with_evicted_tokens():
    gh, gw, rows, pools = _load_worked_example()
    fid = np.array([[r[0] for r in rows]], np.uint32)
    pid = np.array([[r[1] for r in rows]], np.uint16)
    van = np.array([[r[2] for r in rows]])
    for k in (3, 5, 7):
        pooled, ks, _ = oracle.van_pool(van, 1, gh, gw, FORCE[k], pid, fid)
        assert ks[0] == k
        for kk, n, x in pools:
            if kk == k:
                assert pooled[0, n] == pytest.approx(x, rel=1e-15), (k, n)


@pytest.mark.parametrize("k", [3, 5, 7])
@pytest.mark.parametrize("grid", [(5, 7), (3, 2), (14, 14)])
def test_whole_frames_match_torch_avg_pool2d(k, grid):
    torch = pytest.importorskip("torch")
    gh, gw = grid
    f, H = 4, 2
    rng = np.random.default_rng(k * 100 + gh)
    van = rng.lognormal(0.0, 0.5, size=(2 * H, f * gh * gw))
    pooled, ks, _ = oracle.van_pool(van, H, gh, gw, FORCE[k])
    assert list(ks) == [k, k]
    x = torch.from_numpy(van.reshape(2 * H * f, 1, gh, gw))
    ref = torch.nn.functional.avg_pool2d(x, k, stride=1, padding=k // 2,
                                         count_include_pad=False).numpy()
    np.testing.assert_allclose(pooled, ref.reshape(van.shape), rtol=1e-13, atol=0)


def test_pool_size_one_is_identity_and_ids_follow_rows():
    rng = np.random.default_rng(3)
    van = rng.lognormal(size=(2, 60))
    pooled, ks, _ = oracle.van_pool(van, 2, 3, 4, FORCE[1])
    assert ks[0] == 1 and np.array_equal(pooled, van)
    # Explicit ids equal to the derived ones (frame n div p, patch n mod p)
    # give the same pooled values as none at all.
    n = np.arange(60)
    pid = np.tile((n % 12).astype(np.uint16), (2, 1))
    fid = np.tile((n // 12).astype(np.uint32), (2, 1))
    for k in (3, 5, 7):
        a = oracle.van_pool(van, 2, 3, 4, FORCE[k])[0]
        b = oracle.van_pool(van, 2, 3, 4, FORCE[k], pid, fid)[0]
        assert np.array_equal(a, b)


def test_scaling_by_a_power_of_two_is_exact():
    rng = np.random.default_rng(4)
    van = rng.lognormal(0.0, 0.7, size=(4, 5 * 12))
    tau = (0.3, 0.6, 0.9)
    a, ka, ca = oracle.van_pool(van, 2, 3, 4, tau)
    b, kb, cb = oracle.van_pool(van * 8.0, 2, 3, 4, tau)
    assert np.array_equal(ka, kb) and np.array_equal(ca, cb)
    assert np.array_equal(b, a * 8.0)


def test_frames_do_not_mix_and_move_with_their_rows():
    gh, gw = 3, 4
    p = gh * gw
    rng = np.random.default_rng(5)
    van = rng.lognormal(size=(1, 4 * p))
    pid = np.tile(np.arange(p, dtype=np.uint16), (1, 4))
    fid = np.repeat(np.array([[3, 8, 11, 20]], np.uint32), p, axis=1)
    base = oracle.van_pool(van, 1, gh, gw, FORCE[5], pid, fid)[0]
    # Changing one frame's values leaves every other frame's pooled values.
    van2 = van.copy()
    van2[0, p:2 * p] *= 3.0
    other = oracle.van_pool(van2, 1, gh, gw, FORCE[5], pid, fid)[0]
    keep = np.r_[0:p, 2 * p:4 * p]
    assert np.array_equal(other[0, keep], base[0, keep])
    # Reordering whole frames (rows and ids together) reorders the result.
    perm = np.r_[3 * p:4 * p, 0:p, 2 * p:3 * p, p:2 * p]
    moved = oracle.van_pool(van[:, perm], 1, gh, gw, FORCE[5], pid[:, perm], fid[:, perm])[0]
    assert np.array_equal(moved, base[:, perm])


def test_patch_id_outside_the_grid_has_no_pooled_value():
    p = 6
    van = np.arange(1.0, 13.0)[None]
    pid = np.tile(np.arange(p, dtype=np.uint16), (1, 2))
    pid[0, 4] = 40
    fid = np.repeat(np.array([[0, 1]], np.uint32), p, axis=1)
    pooled = oracle.van_pool(van, 1, 2, 3, FORCE[3], pid, fid)[0]
    assert math.isnan(pooled[0, 4])
    assert not np.isnan(np.delete(pooled[0], 4)).any()
    # row 1 (patch 1 at (0,1)) sees patches 0,1,2,3,5 of frame 0 (4 is gone)
    assert pooled[0, 1] == pytest.approx((1 + 2 + 3 + 4 + 6) / 5)


def test_van_all_includes_recent_rows():
    # Pythagorean-triple rows: exact norms 5 * 2^k on every row.
    S, N, D = 2, 12, 4
    V = np.zeros((S, N, D), np.float32)
    V[..., 0] = 3.0 * 2.0 ** (np.arange(N) % 3)
    V[..., 1] = 4.0 * 2.0 ** (np.arange(N) % 3)
    van = oracle.van_all(V, N)
    assert np.array_equal(van, np.tile(5.0 * 2.0 ** (np.arange(N) % 3), (S, 1)))


def test_pooled_pass_reduces_to_the_raw_pass_at_pool_size_one():
    w = synth.CONFIGS["tiny"].scaled(n_kv_heads=2, n_layers=2)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    raw = oracle.compress(K, V, w.n_tokens, w.p, r, w.budget, w.tar_ratio)
    pooled = oracle.compress_pooled(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget,
                                    w.tar_ratio, FORCE[1], w.n_kv_heads)
    assert list(pooled[5]) == [1, 1]
    for a, b in zip(raw, pooled[:4]):
        assert np.array_equal(a, b)
    # frame ids of a fresh cache travel as kept div p
    assert np.array_equal(pooled[4][:, :w.budget], raw[0] // w.p)


def test_pooled_pass_cv_counts_the_recent_frames():
    # Past rows all have VaN 1 and recent rows VaN 3: the layer's CV is
    # non-zero only because the recent frames count (Algorithm 2 takes mu
    # and sigma over the whole layer).
    p, f, D = 4, 8, 4
    N = p * f
    r = oracle.recent_frames(f)
    K = np.random.default_rng(6).standard_normal((1, N, D)).astype(np.float32)
    V = np.zeros((1, N, D), np.float32)
    V[0, :, 0] = 1.0
    V[0, N - r * p:, 0] = 3.0
    frac = r * p / N
    cv = math.sqrt(frac * (1 - frac)) * 2 / (1 + 2 * frac)
    tau = (cv * 0.9, cv * 1.1, cv * 4)      # this CV -> 5; past rows alone (CV 0) -> 7
    out = oracle.compress_pooled(K, V, N, 2, 2, r, 20, 0.5, tau, 1)
    assert list(out[5]) == [5]
    # recent rows scored as 0 instead of 3 would give CV sqrt(frac(1-frac))/(1-frac)
    assert math.sqrt(frac * (1 - frac)) / (1 - frac) < tau[0]


def test_pooled_pass_ranks_pooled_values():
    # Grid 1 x 3, 8 frames, r = 1, alpha = 0, budget 4: the VaN stage takes
    # one past token. Raw VaN peaks at an isolated spike (frame 0, patch 0:
    # 10 beside two zeros); pooled with k = 3 that spike averages to 5, below
    # frame 1's uniform 6, whose lowest row (3) is kept instead of row 0.
    p, f, D = 3, 8, 2
    N = p * f
    K = np.random.default_rng(7).standard_normal((1, N, D)).astype(np.float32)
    V = np.zeros((1, N, D), np.float32)
    V[0, :, 0] = 1.0
    V[0, 0:3, 0] = [10.0, 0.0, 0.0]
    V[0, 3:6, 0] = 6.0
    r = oracle.recent_frames(f)
    assert r == 1
    raw = oracle.compress(K, V, N, p, r, 4, 0.0)[0]
    assert raw[0].tolist() == [0, 21, 22, 23]
    out = oracle.compress_pooled(K, V, N, 1, 3, r, 4, 0.0, FORCE[3], 1)
    assert out[0][0].tolist() == [3, 21, 22, 23]
