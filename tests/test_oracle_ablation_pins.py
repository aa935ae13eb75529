"""Pins for the oracle's ablation variants (Sec. 4 ablation table: "TaR
Reverse", "VaN Reverse", "TaR Frame", "Uniform Select"): hand-worked
selections on the golden example, the frame mean on hand arrays (fresh and
compacted frames), the identities that tie the variants to the plain pass,
and the closed forms of uniform frame sampling. Runs on CPU only."""
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _example():
    K, V = [], []
    with open(os.path.join(GOLDEN, "tar_van_worked_example.txt")) as fh:
        for line in fh:
            f = line.split("#", 1)[0].split()
            if f and f[0] == "K":
                K.append([float(x) for x in f[1:]])
            elif f and f[0] == "V":
                V.append([float(x) for x in f[1:]])
    cases = []
    with open(os.path.join(GOLDEN, "ablation_worked_example.txt")) as fh:
        for line in fh:
            f = line.split("#", 1)[0].split()
            if f and f[0] == "ABLATE":
                cases.append((f[1], int(f[2]), float(f[3]), [int(x) for x in f[4:]]))
    return np.array(K, np.float32)[None], np.array(V, np.float32)[None], cases


def test_worked_example():
    K, V, cases = _example()
    assert len(cases) == 7
    for variant, budget, alpha, want in cases:
        kept = oracle.compress_ablation(K, V, 8, 1, 2, 2, budget, alpha, variant)[0]
        assert kept[0].tolist() == want, (variant, budget, alpha)


def test_frame_mean_hand_arrays():
    t = np.array([[1.0, 3.0, 5.0, 9.0, 100.0, 200.0]])
    np.testing.assert_array_equal(oracle.frame_mean(t, 4, 2), [[2, 2, 7, 7, 100, 200]])  # recent rows kept
    fid = np.array([[4, 4, 6, 6, 6, 9]], np.uint32)
    t = np.array([[1.0, 2.0, 3.0, 4.0, 8.0, 0.0]])
    np.testing.assert_array_equal(oracle.frame_mean(t, 5, 3, fid), [[1.5, 1.5, 5, 5, 5, 0]])


def test_reverse_variants_are_the_plain_pass_on_negated_scores():
    w = synth.CONFIGS["tiny"].scaled(n_kv_heads=3)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    tar, van = oracle.scores(K, V, w.n_tokens, w.p, r)
    for variant, (t, v) in {"tar_reverse": (-tar, van), "van_reverse": (tar, -van)}.items():
        want = oracle.select(t, v, w.n_tokens, w.p, r, w.budget, w.tar_ratio)
        got = oracle.compress_ablation(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget,
                                       w.tar_ratio, variant)[0]
        assert np.array_equal(got, want), variant
    # TaR Frame: the plain selection on frame-mean TaR
    n_past = w.n_tokens - r * w.p
    want = oracle.select(oracle.frame_mean(tar, n_past, w.p), van, w.n_tokens, w.p, r, w.budget,
                         w.tar_ratio)
    got = oracle.compress_ablation(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget,
                                   w.tar_ratio, "tar_frame")[0]
    assert np.array_equal(got, want)


def test_frame_level_tar_keeps_whole_frames_at_alpha_one():
    w = synth.CONFIGS["tiny"].scaled(n_kv_heads=2, budget=16 + 3 * 16)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    kept = oracle.compress_ablation(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget, 1.0,
                                    "tar_frame")[0]
    for s in range(2):
        past = kept[s][kept[s] < w.n_tokens - r * w.p]
        frames, counts = np.unique(past // w.p, return_counts=True)
        assert len(frames) == 3 and np.all(counts == w.p)      # three whole frames


def test_frame_level_tar_needs_frame_ids_with_patch_ids():
    w = synth.CONFIGS["tiny"]
    K, V = synth.host_generate(w)
    pid = np.tile((np.arange(w.n_tokens) % w.p).astype(np.uint16), (w.n_slabs, 1))
    with pytest.raises(ValueError):
        oracle.compress_ablation(K, V, w.n_tokens, w.grid_h, w.grid_w, 1, w.budget, 0.5,
                                 "tar_frame", patch_id=pid)


@pytest.mark.parametrize("F,k,p", [(48, 32, 196), (64, 48, 256), (10, 3, 5), (9, 8, 4), (12, 4, 7),
                                   (7, 1, 3), (100, 37, 2)])
def test_uniform_select_closed_forms(F, k, p):
    """Whole frames, ascending, exactly budget rows; the newest frame always;
    consecutive kept frames floor(F/k) or ceil(F/k) apart; the frames are
    F - 1 - floor(i F / k) for i < k (brute force); every (F/k)-th frame back
    from the newest when k divides F; the oldest frame alone dropped when
    k = F - 1."""
    kept = oracle.uniform_select(2, F * p, p, k * p)
    assert np.array_equal(kept[0], kept[1])
    rows = kept[0]
    assert len(rows) == k * p and np.all(np.diff(rows) > 0)
    frames = rows.reshape(k, p) // p
    assert np.all(frames == frames[:, :1])                         # whole frames
    assert np.array_equal(rows.reshape(k, p) % p, np.tile(np.arange(p), (k, 1)))
    f = frames[:, 0]
    assert f[-1] == F - 1                                          # the newest frame
    gaps = set(np.diff(f).tolist())
    assert gaps <= {F // k, -(-F // k)}
    # brute force: the frames are exactly F - 1 - floor(i F / k), i < k
    assert sorted(f.tolist()) == sorted(F - 1 - (i * F) // k for i in range(k))
    if F % k == 0:
        assert np.array_equal(f, np.arange(F - 1 - (k - 1) * (F // k), F, F // k))
    if k == F - 1:
        assert np.array_equal(f, np.arange(1, F))


def test_uniform_select_reads_no_score():
    """The same indices whatever the keys and values hold; the compacted rows
    are the source rows of those indices."""
    w = synth.CONFIGS["tiny"].scaled(n_kv_heads=3, n_frames=12, budget=5 * 16)
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(w.n_frames)
    got = oracle.compress_ablation(K, V, w.n_tokens, w.grid_h, w.grid_w, r, w.budget, 0.3, "uniform")
    rng = np.random.default_rng(5)
    K2 = rng.standard_normal(K.shape).astype(K.dtype)
    V2 = -3.0 * V
    got2 = oracle.compress_ablation(K2, V2, w.n_tokens, w.grid_h, w.grid_w, r, w.budget, 0.9,
                                    "uniform")
    want = oracle.uniform_select(w.n_slabs, w.n_tokens, w.p, w.budget)
    assert np.array_equal(got[0], want) and np.array_equal(got2[0], want)
    for s in range(w.n_slabs):
        assert np.array_equal(got[1][s, :w.budget], K[s, want[s]])
        assert np.array_equal(got[2][s, :w.budget], V[s, want[s]])
    assert np.array_equal(got[3][:, :w.budget], (want % w.p).astype(np.uint16))
    assert np.array_equal(got[4][:, :w.budget], (want // w.p).astype(np.uint32))


def test_uniform_select_rejects_partial_frames_and_passes_small_caches():
    with pytest.raises(ValueError):
        oracle.uniform_select(1, 40, 4, 10)       # budget not a whole number of frames
    w = synth.CONFIGS["tiny"]
    K, V = synth.host_generate(w)
    kept = oracle.compress_ablation(K, V, w.n_tokens, w.grid_h, w.grid_w, 1, w.n_tokens + 16, 0.5,
                                    "uniform")[0]
    want = list(range(w.n_tokens)) + [-1] * 16
    assert all(row.tolist() == want for row in kept)               # pass-through
