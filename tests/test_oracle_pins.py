"""Pins for the CPU oracle against what the paper and the mathematics fix.

Each test ties the oracle to something other than itself: a hand-worked
example (tests/golden), closed forms of Eq. (tar) and of the L2 norm,
invariances, special cases that reduce to a library routine, and brute force
over every subset on tiny inputs. Runs on CPU only.
"""
import itertools
import math
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load_worked_example():
    meta, K, V, tar, van, sel = {}, [], [], {}, {}, []
    with open(os.path.join(GOLDEN, "tar_van_worked_example.txt")) as fh:
        for line in fh:
            line = line.split("#", 1)[0].split()
            if not line:
                continue
            tag, rest = line[0], line[1:]
            if tag in ("D", "P", "N", "R"):
                meta[tag] = int(rest[0])
            elif tag == "K":
                K.append([float(x) for x in rest])
            elif tag == "V":
                V.append([float(x) for x in rest])
            elif tag == "TAR":
                tar[int(rest[0])] = float(rest[1])
            elif tag == "VAN":
                van[int(rest[0])] = float(rest[1])
            elif tag == "SELECT":
                sel.append((int(rest[0]), float(rest[1]), [int(x) for x in rest[2:]]))
    K = np.array(K, np.float32)[None]
    V = np.array(V, np.float32)[None]
    return meta, K, V, tar, van, sel


def test_worked_example_scores():
    meta, K, V, tar_x, van_x, _ = _load_worked_example()
    tar, van = oracle.scores(K, V, meta["N"], meta["P"], meta["R"])
    for n, x in tar_x.items():
        assert tar[0, n] == pytest.approx(x, abs=1e-15)
    for n, x in van_x.items():
        assert van[0, n] == x  # exact: integer or dyadic norms


def test_worked_example_selection():
    meta, K, V, _, _, sel = _load_worked_example()
    tar, van = oracle.scores(K, V, meta["N"], meta["P"], meta["R"])
    for budget, alpha, expect in sel:
        kept = oracle.select(tar, van, meta["N"], meta["P"], meta["R"], budget, alpha)
        assert kept[0].tolist() == expect, (budget, alpha)


def _rand_keys(rng, S, f, p, D):
    return rng.standard_normal((S, f * p, D)).astype(np.float32)


@pytest.mark.parametrize("r", [1, 2, 3])
def test_identical_frames_give_minus_one(r):
    """Eq. (tar): identical patch-aligned keys have cosine 1, so s_TaR = -1."""
    rng = np.random.default_rng(1)
    S, f, p, D = 2, 6, 5, 16
    frame = rng.standard_normal((S, 1, p, D)).astype(np.float32)
    K = np.repeat(frame, f, axis=1).reshape(S, f * p, D)
    V = _rand_keys(rng, S, f, p, D)
    tar, _ = oracle.scores(K, V, f * p, p, r)
    past = (f - r) * p
    assert np.allclose(tar[:, :past], -1.0, atol=1e-12, rtol=0)
    assert np.all(tar[:, past:] == 0.0)


def test_orthogonal_and_negated_keys():
    """cos = 0 for orthogonal keys (s = 0); cos = -1 for negated keys (s = +1)."""
    D, p, f, r = 4, 2, 3, 1
    K = np.zeros((1, f * p, D), np.float32)
    K[0, 0] = [1, 0, 0, 0]          # past frame0 patch0
    K[0, 1] = [0, 0, 2, 0]          # past frame0 patch1
    K[0, 2] = [0, 5, 0, 0]          # past frame1 patch0
    K[0, 3] = [0, 0, 1, 1]          # past frame1 patch1
    K[0, 4] = [0, 3, 0, 0]          # recent patch0
    K[0, 5] = [0, 0, -7, 0]         # recent patch1
    V = np.ones_like(K)
    tar, _ = oracle.scores(K, V, f * p, p, r)
    assert tar[0, 0] == 0.0                      # e1 vs e2: orthogonal
    assert tar[0, 1] == 1.0                      # e3 vs -e3: negated
    assert tar[0, 2] == -1.0                     # e2 vs e2: identical direction
    assert tar[0, 3] == pytest.approx(1 / math.sqrt(2), abs=1e-15)


def test_scale_invariance():
    """TaR uses l2-normalised keys: positive rescaling of any key changes nothing."""
    rng = np.random.default_rng(2)
    S, f, p, D, r = 3, 8, 4, 32, 2
    K = _rand_keys(rng, S, f, p, D)
    V = _rand_keys(rng, S, f, p, D)
    tar0, van0 = oracle.scores(K, V, f * p, p, r)
    scale = rng.uniform(0.25, 4.0, size=(S, f * p, 1)).astype(np.float32)
    tar1, van1 = oracle.scores(K * scale, V, f * p, p, r)
    assert np.allclose(tar0, tar1, atol=1e-6, rtol=0)  # fp32 inputs rescaled with rounding
    pow2 = np.float32(2.0) ** rng.integers(-8, 8, size=(S, f * p, 1)).astype(np.float32)
    tar2, _ = oracle.scores(K * pow2, V, f * p, p, r)
    assert np.allclose(tar0, tar2, atol=1e-14, rtol=0)  # exact rescaling
    assert np.array_equal(van0, van1)


def test_r1_is_cosine_to_latest_frame():
    """With r = 1 the mean over recent frames is the latest frame alone."""
    rng = np.random.default_rng(3)
    S, f, p, D = 2, 5, 3, 8
    K = _rand_keys(rng, S, f, p, D).astype(np.float64).astype(np.float32)
    V = _rand_keys(rng, S, f, p, D)
    tar, _ = oracle.scores(K, V, f * p, p, 1)
    Kd = K.astype(np.float64)
    for s in range(S):
        for n in range((f - 1) * p):
            a, b = Kd[s, n], Kd[s, (f - 1) * p + n % p]
            c = np.dot(a, b) / (np.linalg.norm(a) * np.linalg.norm(b))
            assert tar[s, n] == pytest.approx(-c, abs=1e-13)


def test_recent_frame_order_irrelevant_and_all_used():
    """The r recent frames enter symmetrically; each of them contributes 1/r."""
    rng = np.random.default_rng(4)
    S, f, p, D, r = 1, 6, 3, 8, 3
    K = _rand_keys(rng, S, f, p, D)
    V = _rand_keys(rng, S, f, p, D)
    tar0, _ = oracle.scores(K, V, f * p, p, r)
    K2 = K.copy().reshape(S, f, p, D)
    K2[:, f - r:] = K2[:, f - r:][:, ::-1]  # reverse the recent frames
    tar1, _ = oracle.scores(K2.reshape(S, f * p, D), V, f * p, p, r)
    assert np.allclose(tar0, tar1, atol=1e-14, rtol=0)
    # Replacing one recent frame by the past token's own direction raises its
    # cosine to exactly 1, so s_TaR drops by (1 - cos_old)/r.
    n, q = 1, 1
    K3 = K.copy().reshape(S, f, p, D)
    old = K3[0, f - 1, q].astype(np.float64)
    k_n = K3.reshape(S, f * p, D)[0, n].astype(np.float64)
    cos_old = old @ k_n / (np.linalg.norm(old) * np.linalg.norm(k_n))
    K3[0, f - 1, q] = K3.reshape(S, f * p, D)[0, n] * 2.0
    tar3, _ = oracle.scores(K3.reshape(S, f * p, D), V, f * p, p, r)
    assert tar3[0, n] == pytest.approx(tar0[0, n] - (1.0 - cos_old) / r, abs=1e-12)


def test_van_exact_norms():
    """Sec. 3.2: VaN = ||v||_2; Pythagorean triples scaled by 2^k are exact."""
    D, p, f, r = 8, 4, 3, 1
    V = np.zeros((1, f * p, D), np.float32)
    triples = [(3, 4, 0, 5), (5, 12, 0, 13), (8, 15, 0, 17), (1, 2, 2, 3)]
    expect = []
    for n in range(f * p):
        a, b, c, h = triples[n % 4]
        k = (n % 7) - 3
        V[0, n, n % 3] = a * 2.0 ** k
        V[0, n, 3 + (n % 2)] = b * 2.0 ** k
        V[0, n, 6] = c * 2.0 ** k
        expect.append(h * 2.0 ** k)
    K = np.random.default_rng(5).standard_normal(V.shape).astype(np.float32)
    _, van = oracle.scores(K, V, f * p, p, r)
    past = (f - r) * p
    assert van[0, :past].tolist() == expect[:past]


def _to_bf16_bits(x):
    """Round-to-nearest-even fp32 -> bf16 bit patterns (numpy, host)."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    return ((u + 0x7FFF + lsb) >> 16).astype(np.uint16)


def test_bf16_inputs_are_widened_exactly():
    """bf16 bit patterns 0x4040 = 3.0 and 0x4080 = 4.0 give VaN exactly 5."""
    D, p, f, r = 2, 1, 2, 1
    V = np.array([[[0x4040, 0x4080], [0x3F80, 0x0000]]], np.uint16)
    K = np.array([[[0x3F80, 0x0000], [0x0000, 0x3F80]]], np.uint16)  # e1 past, e2 recent
    tar, van = oracle.scores(K, V, f * p, p, r)
    assert van[0, 0] == 5.0 and tar[0, 0] == 0.0
    x = np.array([1.0, 3.0, -2.5, 1.00390625], np.float32)  # last one is a bf16 tie
    assert _to_bf16_bits(x).tolist() == [0x3F80, 0x4040, 0xC020, 0x3F80]


def test_patch_ids_are_followed():
    """Past tokens are compared with the recent frames at their own patch id:
    permuting past rows together with their ids permutes the scores."""
    rng = np.random.default_rng(6)
    S, f, p, D, r = 2, 5, 4, 16, 1
    K = _rand_keys(rng, S, f, p, D)
    V = _rand_keys(rng, S, f, p, D)
    N = f * p
    past = (f - r) * p
    tar0, van0 = oracle.scores(K, V, N, p, r)
    perm = rng.permutation(past)
    K2, V2 = K.copy(), V.copy()
    K2[:, :past] = K[:, perm]
    V2[:, :past] = V[:, perm]
    pid = np.tile((np.arange(N) % p).astype(np.uint16), (S, 1))
    pid[:, :past] = (perm % p).astype(np.uint16)
    tar1, van1 = oracle.scores(K2, V2, N, p, r, patch_id=pid)
    assert np.array_equal(tar1[:, :past], tar0[:, perm])
    assert np.array_equal(van1[:, :past], van0[:, perm])
    tar_wrong, _ = oracle.scores(K2, V2, N, p, r)  # ignoring the ids changes TaR
    assert not np.allclose(tar_wrong[:, :past], tar0[:, perm])


@pytest.mark.parametrize("f,expect", [(8, 1), (48, 6), (64, 8), (128, 16), (4, 1), (12, 2)])
def test_recent_frames_default(f, expect):
    """Appendix B.2: r = 0.125 f (rounded, at least one frame)."""
    assert oracle.recent_frames(f) == expect
    assert oracle.recent_frames(f, 3) == 3


@pytest.mark.parametrize("args,expect", [
    ((9408, 196, 6, 6272, 0.5), (1176, 1960, 3136)),
    ((16384, 256, 8, 12288, 0.3), (2048, 1638, 8602)),  # floor(0.3*12288) = 3686
    ((128, 16, 1, 48, 0.5), (16, 8, 24)),
    ((32768, 256, 16, 24576, 0.5), (4096, 8192, 12288)),
    ((100, 10, 2, 50, 0.0), (20, 0, 30)),     # alpha = 0: VaN only (Tab. A1)
    ((100, 10, 2, 50, 1.0), (20, 30, 0)),     # alpha = 1: TaR only (Tab. A1)
    ((100, 10, 2, 50, 0.3), (20, 0, 30)),     # floor(15) < rp: no TaR picks
])
def test_budget_split(args, expect):
    """Sec. 3.3 / Algorithm 1: alpha|C| for TaR incl. the recent frames, rest VaN."""
    assert oracle.budget_split(*args) == expect
    assert sum(expect) == args[3]


def test_budget_split_passthrough_and_errors():
    assert oracle.budget_split(48, 16, 1, 48, 0.5) is None      # N == C
    assert oracle.budget_split(30, 10, 1, 48, 0.5) is None      # N < C
    with pytest.raises(ValueError):
        oracle.budget_split(100, 10, 5, 50, 0.5)                # rp == C
    with pytest.raises(ValueError):
        oracle.budget_split(100, 10, 2, 50, 1.5)


def _topk_lexsort(score, cand, k):
    """Library reference: the k best of cand by (score desc, index asc)."""
    cand = np.asarray(cand)
    order = np.lexsort((cand, -score[cand]))
    return set(cand[order[:k]].tolist())


def _check_invariants(kept, N, rp, budget):
    for row in kept:
        assert len(row) == budget
        assert np.all(np.diff(row) > 0)                       # ascending, distinct
        assert set(range(N - rp, N)) <= set(row.tolist())     # recent frames kept
        assert row.min() >= 0 and row.max() < N


@pytest.mark.parametrize("seed", range(5))
def test_selection_matches_lexsort(seed):
    """TaR top-k over past tokens, then VaN top over the rest, ties to lower index."""
    rng = np.random.default_rng(seed)
    S, f, p, r, budget = 3, 10, 7, 2, 40
    N = f * p
    for alpha in (0.0, 0.3, 0.5, 0.8, 1.0):
        tar = rng.integers(-4, 4, size=(S, N)).astype(np.float64) / 4  # many ties
        van = rng.integers(0, 6, size=(S, N)).astype(np.float64)
        kept = oracle.select(tar, van, N, p, r, budget, alpha)
        rp, n_tar, n_van = oracle.budget_split(N, p, r, budget, alpha)
        _check_invariants(kept, N, rp, budget)
        past = np.arange(N - rp)
        for s in range(S):
            t_set = _topk_lexsort(tar[s], past, n_tar)
            rest = np.array(sorted(set(past.tolist()) - t_set), dtype=np.int64)
            v_set = _topk_lexsort(van[s], rest, n_van)
            expect = sorted(t_set | v_set | set(range(N - rp, N)))
            assert kept[s].tolist() == expect


def test_selection_bruteforce_subsets():
    """Every subset of the right size is tried; exactly one dominates under
    (score desc, index asc) and it is the oracle's, for both stages."""
    rng = np.random.default_rng(7)
    p, f, r, budget, alpha = 2, 8, 1, 9, 0.6  # N=16, rp=2, n_past=14
    N = p * f
    rp, n_tar, n_van = oracle.budget_split(N, p, r, budget, alpha)
    assert (rp, n_tar, n_van) == (2, 3, 4)
    for trial in range(4):
        tar = np.round(rng.standard_normal((1, N)), 1)
        van = np.round(np.abs(rng.standard_normal((1, N))), 1)
        kept = set(oracle.select(tar, van, N, p, r, budget, alpha)[0].tolist())
        past = list(range(N - rp))

        def better(sc, a, b):
            return sc[a] > sc[b] or (sc[a] == sc[b] and a < b)

        def dominating(sc, cand, k):
            winners = []
            for sub in itertools.combinations(cand, k):
                out = [x for x in cand if x not in sub]
                if all(better(sc, a, b) for a in sub for b in out):
                    winners.append(set(sub))
            assert len(winners) == 1
            return winners[0]

        t_set = dominating(tar[0], past, n_tar)
        rest = [x for x in past if x not in t_set]
        v_set = dominating(van[0], rest, n_van)
        assert kept == t_set | v_set | set(range(N - rp, N))


def test_alpha_extremes_reduce_to_single_metric():
    """alpha = 0 keeps past tokens by VaN alone; alpha = 1 by TaR alone (Tab. A1)."""
    rng = np.random.default_rng(8)
    S, f, p, r, budget = 2, 12, 5, 1, 30
    N = f * p
    K = _rand_keys(rng, S, f, p, 8)
    V = _rand_keys(rng, S, f, p, 8)
    tar, van = oracle.scores(K, V, N, p, r)
    past = np.arange(N - r * p)
    k0 = oracle.select(tar, van, N, p, r, budget, 0.0)
    k1 = oracle.select(tar, van, N, p, r, budget, 1.0)
    for s in range(S):
        assert set(k0[s].tolist()) - set(range(N - p, N)) == _topk_lexsort(van[s], past, budget - p)
        assert set(k1[s].tolist()) - set(range(N - p, N)) == _topk_lexsort(tar[s], past, budget - p)


def test_nan_ranks_lowest():
    N, p, r, budget = 8, 1, 1, 4
    tar = np.array([[np.nan, 1.0, np.nan, -5.0, 0.5, 2.0, np.nan, 0.0]])
    van = np.zeros_like(tar)
    kept = oracle.select(tar, van, N, p, r, budget, 1.0)  # 3 TaR picks + 1 recent
    assert kept[0].tolist() == [1, 4, 5, 7]


def test_passthrough_and_identity():
    """A cache at or below the budget is not compressed (Algorithm 1 trigger)."""
    rng = np.random.default_rng(9)
    S, f, p, D = 2, 3, 4, 8
    N = f * p
    K = _rand_keys(rng, S, f, p, D)
    V = _rand_keys(rng, S, f, p, D)
    tar = np.zeros((S, N))
    kept = oracle.select(tar, tar, N, p, 1, N + 5, 0.5)
    assert kept.tolist() == [list(range(N)) + [-1] * 5] * S
    kept2, kd, vd, _ = oracle.compress(K, V, N, p, 1, N, 0.5)
    assert kept2.tolist() == [list(range(N))] * S
    assert not kd.any() and not vd.any()  # nothing is copied in pass-through


def test_gather_bytes_and_patch_ids():
    rng = np.random.default_rng(10)
    S, cap, D, budget = 3, 20, 6, 7
    src = rng.integers(0, 65535, size=(S, cap, D)).astype(np.uint16)
    kept = np.stack([np.sort(rng.choice(cap, budget, replace=False)) for _ in range(S)]).astype(np.int32)
    dst = oracle.gather(src, kept)
    for s in range(S):
        assert np.array_equal(dst[s, :budget], src[s, kept[s]])
        assert not dst[s, budget:].any()
    pid_src = rng.integers(0, 5, size=(S, cap)).astype(np.uint16)
    pd = oracle.gather_patch(pid_src, kept, 5, cap, cap)
    pd0 = oracle.gather_patch(None, kept, 5, cap, cap)
    for s in range(S):
        assert np.array_equal(pd[s, :budget], pid_src[s, kept[s]])
        assert np.array_equal(pd0[s, :budget], kept[s] % 5)


def test_compress_end_to_end_small():
    """scores -> select -> gather agree with the stage functions called one by one."""
    rng = np.random.default_rng(11)
    S, f, p, D, r, budget, alpha = 2, 8, 16, 64, 1, 48, 0.5
    N = f * p
    K = _rand_keys(rng, S, f, p, D)
    V = _rand_keys(rng, S, f, p, D)
    kept, kd, vd, pd = oracle.compress(K, V, N, p, r, budget, alpha)
    tar, van = oracle.scores(K, V, N, p, r)
    assert np.array_equal(kept, oracle.select(tar, van, N, p, r, budget, alpha))
    for s in range(S):
        assert np.array_equal(kd[s, :budget], K[s, kept[s]])
        assert np.array_equal(vd[s, :budget], V[s, kept[s]])
        assert np.array_equal(pd[s, :budget], kept[s] % p)


def test_boundary_gaps():
    N, p, r, budget = 6, 1, 1, 3
    tar = np.array([[0.9, 0.5, 0.7, 0.1, 0.2, 0.0]])   # past = rows 0..4
    van = np.array([[1.0, 8.0, 2.0, 4.0, 3.0, 0.0]])
    kept, gaps = oracle.select(tar, van, N, p, r, budget, 0.67, with_gaps=True)
    # floor(0.67*3)=2 -> 1 TaR pick (row0, next best 0.7): gap 0.2;
    # VaN picks 1 of {1,2,3,4}: row1 (8), next 4 -> relative gap 0.5.
    assert kept[0].tolist() == [0, 1, 5]
    assert gaps[0, 0] == pytest.approx(0.2, abs=1e-15)
    assert gaps[0, 1] == pytest.approx(0.5, abs=1e-15)
