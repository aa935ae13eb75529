"""GPU-vs-oracle comparison rules shared by the GPU tests.

Acceptance (fp32 GPU arithmetic against the fp64 oracle):
  * scores: TaR |g - o| <= 1e-5 max(|o|, 1)   (TaR lies in [-1, 1]);
            VaN |g - o| <= 1e-5 |o|;
  * indices: the GPU's selection must equal the exact selection on its own
    fp32 scores (checked bit for bit), and its kept set must equal the
    oracle's, except where an oracle stage's boundary gap is below 1e-5
    (absolute for TaR, relative for VaN); then only tokens whose oracle score
    lies within 1e-5 of that boundary may differ, and the VaN stage is judged
    against the oracle's VaN choice among the tokens the GPU's TaR stage left;
  * K/V bytes: exact given the GPU's indices.
"""
from __future__ import annotations

import numpy as np

import oracle

TOL = 1e-5


def assert_scores_close(g_tar, g_van, o_tar, o_van, n_past):
    g_tar = np.asarray(g_tar, np.float64)[:, :n_past]
    g_van = np.asarray(g_van, np.float64)[:, :n_past]
    o_tar = o_tar[:, :n_past]
    o_van = o_van[:, :n_past]
    err_t = np.abs(g_tar - o_tar) / np.maximum(np.abs(o_tar), 1.0)
    err_v = np.abs(g_van - o_van) / np.maximum(np.abs(o_van), 1e-30)
    assert np.all(np.isfinite(g_tar)) and np.all(np.isfinite(g_van))
    assert err_t.max(initial=0.0) <= TOL, f"TaR error {err_t.max():.3g} at {np.unravel_index(err_t.argmax(), err_t.shape)}"
    assert err_v.max(initial=0.0) <= TOL, f"VaN error {err_v.max():.3g} at {np.unravel_index(err_v.argmax(), err_v.shape)}"
    return float(err_t.max(initial=0.0)), float(err_v.max(initial=0.0))


def _topk(score, cand, k):
    cand = np.asarray(cand, np.int64)
    if k <= 0:
        return set()
    order = np.lexsort((cand, -score[cand]))
    return set(cand[order[:k]].tolist())


def _boundary_window(score, cand, k, relative):
    """(lo, hi) score window around the k-th boundary, or None if the gap >= TOL."""
    cand = np.asarray(cand, np.int64)
    if k <= 0 or k >= len(cand):
        return None
    order = cand[np.lexsort((cand, -score[cand]))]
    a, b = score[order[k - 1]], score[order[k]]
    gap = abs(a - b) / (max(abs(a), 1e-300) if relative else 1.0)
    if gap >= TOL:
        return None
    tol = TOL * (max(abs(a), 1e-300) if relative else 1.0)
    return b - tol, a + tol


def _check_stage(name, s, got, want, score, cand, k, relative):
    if got == want:
        return 0
    win = _boundary_window(score, cand, k, relative)
    assert win is not None, f"slab {s}: {name} set differs with a boundary gap >= {TOL}"
    diff = got ^ want
    bad = [n for n in diff if not (win[0] <= score[n] <= win[1])]
    assert not bad, f"slab {s}: {name} differs outside the boundary window: {bad[:8]}"
    return len(diff)


def assert_selection_matches(kept_g, g_tar, g_van, o_tar, o_van, N, p, r, budget, alpha):
    """kept_g: GPU indices [S, budget]; g_*: GPU fp32 scores; o_*: oracle fp64."""
    kept_g = np.asarray(kept_g)
    alpha_f = float(np.float32(alpha))  # the library takes alpha as fp32
    split = oracle.budget_split(N, p, r, budget, alpha_f)
    S = kept_g.shape[0]
    if split is None:
        want = np.tile(np.array(list(range(N)) + [-1] * (budget - N), np.int32), (S, 1))
        assert np.array_equal(kept_g, want)
        return 0
    rp, n_tar, n_van = split
    n_past = N - rp
    # (1) the GPU picks exactly what the definition picks on its own scores
    exact = oracle.select(np.asarray(g_tar, np.float64), np.asarray(g_van, np.float64),
                          N, p, r, budget, alpha_f)
    mism = np.nonzero(~np.all(exact == kept_g, axis=1))[0]
    assert mism.size == 0, f"selection differs from the exact rule on GPU scores in slabs {mism[:8].tolist()}"
    # (2) against the fp64 oracle with the boundary-gap rule
    past = np.arange(n_past)
    recent = set(range(n_past, N))
    n_diff = 0
    for s in range(S):
        got = set(kept_g[s].tolist())
        assert recent <= got and len(got) == budget
        gt = np.asarray(g_tar[s], np.float64)
        t_g = _topk(gt, past, n_tar)
        t_o = _topk(o_tar[s], past, n_tar)
        n_diff += _check_stage("TaR", s, t_g, t_o, o_tar[s], past, n_tar, relative=False)
        rest = np.array(sorted(set(past.tolist()) - t_g), np.int64)
        v_g = got - t_g - recent
        v_o = _topk(o_van[s], rest, n_van)
        n_diff += _check_stage("VaN", s, v_g, v_o, o_van[s], rest, n_van, relative=True)
    return n_diff


def assert_gather_exact(src, dst, kept, budget):
    """dst rows 0..budget-1 equal src rows kept (byte arrays [S, cap, D])."""
    S = kept.shape[0]
    for s in range(S):
        idx = kept[s]
        assert np.array_equal(dst[s, :budget], src[s, idx]), f"slab {s}: compacted rows differ"


INF = float("inf")
FORCE_POOL = {7: (INF, INF, INF), 5: (0.0, INF, INF), 3: (0.0, 0.0, INF), 1: (0.0, 0.0, 0.0)}


def pooled_reference(van_all_o, n_heads, gh, gw, tau, ks_gpu, pid=None, fid=None):
    """Oracle pooled VaN for layer-adaptive pooling, checked against the GPU's
    per-layer pool sizes. The pool size is an integer decided by a floating
    CV: it must equal the oracle's, except where the oracle's CV lies within
    TOL (relative) of a threshold; there the GPU's size is accepted and the
    oracle pools with it. Returns (pooled [S, N], oracle sizes, oracle CVs)."""
    pooled, ks, cv = oracle.van_pool(van_all_o, n_heads, gh, gw, tau, pid, fid)
    for layer in range(len(ks)):
        kg = int(ks_gpu[layer])
        if kg == ks[layer]:
            continue
        near = any(abs(cv[layer] - t) <= TOL * max(abs(t), 1e-30) for t in tau)
        assert near, f"layer {layer}: pool size {kg} vs oracle {ks[layer]} (CV {cv[layer]:.9g})"
        sl = slice(layer * n_heads, (layer + 1) * n_heads)
        sub_p = None if pid is None else pid[sl]
        sub_f = None if fid is None else fid[sl]
        pooled[sl] = oracle.van_pool(van_all_o[sl], n_heads, gh, gw, FORCE_POOL[kg], sub_p, sub_f)[0]
    return pooled, ks, cv


def assert_pooled_close(g, o, rows=None):
    """Pooled VaN: |g - o| <= TOL |o| (NaN exactly where the oracle has NaN)."""
    g = np.asarray(g, np.float64)
    if rows is not None:
        g, o = g[:, :rows], o[:, :rows]
    nan_o = np.isnan(o)
    assert np.array_equal(np.isnan(g), nan_o), "NaN positions differ"
    err = np.abs(g - o)[~nan_o] / np.maximum(np.abs(o[~nan_o]), 1e-30)
    assert err.max(initial=0.0) <= TOL, f"pooled VaN error {err.max():.3g}"
    return float(err.max(initial=0.0))
