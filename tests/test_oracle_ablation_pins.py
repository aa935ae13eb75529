"""Pins for the oracle's ablation variants (Sec. 4 ablation table: "TaR
Reverse", "VaN Reverse", "TaR Frame"): hand-worked selections on the golden
example, the frame mean on hand arrays (fresh and compacted frames), and the
identities that tie the variants to the plain pass. Runs on CPU only."""
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
    assert len(cases) == 4
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
