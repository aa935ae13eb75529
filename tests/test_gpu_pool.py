"""GPU parity of layer-adaptive VaN pooling (Sec. 3.2 "Layer-wise Adaptive
Pooling"; Algorithm 2) against the CPU oracle, through the C ABI:

- `ipv_van_pool` on VaN values both sides read as the same fp32 numbers;
- the whole pass with `van_pool` on, for fresh and compacted caches (patch
  and frame ids);
- the LLaVA-shaped pooled workload at full size, on sampled whole layers.

Rules: parity.py (scores 1e-5; pool sizes exact unless the oracle's CV is
within 1e-5 of a threshold; indices exact up to boundary ties; bytes exact).
"""
import numpy as np
import pytest

import oracle
import synth
from parity import (FORCE_POOL, assert_gather_exact, assert_pooled_close, assert_scores_close,
                    assert_selection_matches, pooled_reference)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2506_15745_gb300 import ipv  # noqa: E402
from paper_2506_15745_gb300.cache import PingPongCache  # noqa: E402


def to_np(t):
    t = t.contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    if t.dtype == torch.int16:
        return t.cpu().numpy().view(np.uint16)
    if t.dtype == torch.int32:
        return t.cpu().numpy()
    return t.cpu().numpy()


def to_dev(a, dtype):
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.fixture(autouse=True)
def _shutdown_after():
    yield
    torch.cuda.synchronize()
    ipv.shutdown()


def spread_tau(cvs, tau):
    """Move each threshold to the midpoint of the two layer CVs around it, so
    that no layer's pool size hangs on rounding."""
    c = np.sort(np.asarray(cvs))
    out = []
    for t in tau:
        i = np.searchsorted(c, t)
        lo = c[i - 1] if i > 0 else t - 1.0
        hi = c[i] if i < len(c) else t + 1.0
        out.append(float(np.float32(0.5 * (lo + hi))))
    return tuple(out)


# ------------------------------------------------------------ the pooling step alone
def _van_case(L, H, gh, gw, f, sigmas, seed):
    rng = np.random.default_rng(seed)
    van = np.concatenate([rng.lognormal(0.0, sigmas[l % len(sigmas)], size=(H, f * gh * gw))
                          for l in range(L)]).astype(np.float32)
    return van


def _run_van_pool(van32, L, H, gh, gw, tau, pid=None, fid=None):
    S, N = van32.shape
    van_d = torch.from_numpy(van32).cuda()
    out = torch.full((S, N), -5.0, dtype=torch.float32, device="cuda")
    ks = torch.full((L,), -1, dtype=torch.int32, device="cuda")
    pid_d = None if pid is None else torch.from_numpy(pid.view(np.int16)).cuda()
    fid_d = None if fid is None else torch.from_numpy(fid.view(np.int32)).cuda()
    ipv.van_pool(van_d, L, H, N, gh, gw, tau, out, ks, pid_d, fid_d,
                 0 if pid is None else pid.shape[1])
    torch.cuda.synchronize()
    return out.cpu().numpy(), ks.cpu().numpy()


@pytest.mark.parametrize("gh,gw,f,H", [(5, 7, 6, 2), (14, 14, 12, 4), (3, 3, 5, 1), (1, 9, 4, 3),
                                       (16, 16, 4, 2)])
def test_van_pool_whole_frames(gh, gw, f, H):
    L = 4
    ipv.init(device=0, dtype="bf16", max_head_dim=64, max_frame_tokens=gh * gw,
             max_slabs=L * H, token_capacity=f * gh * gw, van_pool=True, cv_tau=(0.3, 0.9, 3.0))
    van = _van_case(L, H, gh, gw, f, (0.1, 0.5, 1.0, 2.0), seed=gh * 100 + gw)
    cv = np.sort(oracle.van_pool(van.astype(np.float64), H, gh, gw, (0, 0, 0))[2])
    tau = tuple(float(np.float32(0.5 * (cv[i] + cv[i + 1]))) for i in range(3))
    g, ks = _run_van_pool(van, L, H, gh, gw, tau)
    o, ko, _ = pooled_reference(van.astype(np.float64), H, gh, gw, tau, ks)
    assert sorted(set(ko.tolist())) == [1, 3, 5, 7]          # all four pool sizes exercised
    assert np.array_equal(ks, ko)
    assert_pooled_close(g, o)


@pytest.mark.parametrize("k", [7, 5, 3, 1])
def test_van_pool_compacted_rows_with_ids(k):
    """Frames that lost tokens in earlier passes (random survivors, some
    frames down to one token), rows in (frame, patch) order, a row stride
    above n_tokens, and one row whose patch id lies outside the grid."""
    gh, gw, H, L = 14, 14, 2, 2
    p = gh * gw
    rng = np.random.default_rng(k)
    S = L * H
    rows_pid, rows_fid = [], []
    for s in range(S):
        pid, fid = [], []
        for t in range(40):
            keep = rng.random() < 0.85
            n_keep = int(rng.integers(1, p + 1)) if keep else 1
            sel = np.sort(rng.choice(p, size=n_keep, replace=False))
            pid.extend(sel.tolist())
            fid.extend([3 * t + s] * n_keep)
        rows_pid.append(pid)
        rows_fid.append(fid)
    N = min(len(x) for x in rows_pid)
    stride = N + 13
    pid = np.zeros((S, stride), np.uint16)
    fid = np.zeros((S, stride), np.uint32)
    for s in range(S):
        pid[s, :N] = rows_pid[s][:N]
        fid[s, :N] = rows_fid[s][:N]
    pid[1, N // 2] = p + 5                                       # no grid position
    van = rng.lognormal(0.0, 0.6, size=(S, N)).astype(np.float32)
    ipv.init(device=0, dtype="bf16", max_head_dim=64, max_frame_tokens=p, max_slabs=S,
             token_capacity=stride, van_pool=True, cv_tau=(0.3, 0.9, 3.0))
    g, ks = _run_van_pool(van, L, H, gh, gw, FORCE_POOL[k], pid, fid)
    o, ko, _ = pooled_reference(van.astype(np.float64), H, gh, gw, FORCE_POOL[k], ks, pid, fid)
    assert list(ks) == [k] * L and list(ko) == [k] * L
    assert_pooled_close(g, o)
    if k > 1:
        assert np.isnan(g[1, N // 2])


@pytest.mark.parametrize("k", [7, 3])
def test_van_pool_compacted_many_tiles(k):
    """A streamed cache's shape: mostly frames of 1-10 surviving tokens, some
    whole frames, 16x16 grid, 16000 rows per slab (more rows than one
    shared-memory staging tile holds)."""
    gh = gw = 16
    p = gh * gw
    H, L = 2, 1
    rng = np.random.default_rng(40 + k)
    N = 16000
    pid = np.zeros((H, N), np.uint16)
    fid = np.zeros((H, N), np.uint32)
    for s in range(H):
        rows, t = 0, 0
        while rows < N:
            n_keep = p if rng.random() < 0.03 else int(rng.integers(1, 11))
            n_keep = min(n_keep, N - rows)
            sel = np.sort(rng.choice(p, size=n_keep, replace=False))
            pid[s, rows:rows + n_keep] = sel
            fid[s, rows:rows + n_keep] = 5 * t + 1
            rows += n_keep
            t += 1
    van = rng.lognormal(0.0, 0.5, size=(H, N)).astype(np.float32)
    ipv.init(device=0, dtype="bf16", max_head_dim=64, max_frame_tokens=p, max_slabs=H,
             token_capacity=N, van_pool=True, cv_tau=(0.3, 0.9, 3.0))
    g, ks = _run_van_pool(van, L, H, gh, gw, FORCE_POOL[k], pid, fid)
    o, _, _ = pooled_reference(van.astype(np.float64), H, gh, gw, FORCE_POOL[k], ks, pid, fid)
    assert list(ks) == [k]
    assert_pooled_close(g, o)


@pytest.mark.parametrize("gh,gw", [(14, 14), (20, 20), (9, 31)])
@pytest.mark.parametrize("k", [7, 5, 3])
def test_van_pool_large_frames(gh, gw, k):
    """Frames of 33 rows up to whole frames, the ones pooled on a per-warp map.
    At 196 cells each frame goes the way that takes fewer reads (token windows
    or separable sums); at 400 and 279 cells (more than 8 cells per lane) every
    such frame takes the token windows. Frame sizes sweep the point where the
    two ways cost the same for each pool size."""
    p = gh * gw
    H, L = 2, 1
    rng = np.random.default_rng(7 * k + gh)
    sizes = [33, 34, 40, 42, 43, 50, 68, 69, 100, 163, 164, p - 1, p, 37, p, 60]
    sizes = [n for n in sizes if 33 <= n <= p]
    pid_rows, fid_rows = [], []
    for t, n in enumerate(sizes):
        sel = np.sort(rng.choice(p, size=n, replace=False))
        pid_rows.extend(sel.tolist())
        fid_rows.extend([2 * t + 1] * n)
    N = len(pid_rows)
    pid = np.tile(np.array(pid_rows, np.uint16), (H, 1))
    fid = np.tile(np.array(fid_rows, np.uint32), (H, 1))
    van = rng.lognormal(0.0, 0.7, size=(H, N)).astype(np.float32)
    ipv.init(device=0, dtype="bf16", max_head_dim=64, max_frame_tokens=p, max_slabs=H,
             token_capacity=N, van_pool=True, cv_tau=(0.3, 0.9, 3.0))
    g, ks = _run_van_pool(van, L, H, gh, gw, FORCE_POOL[k], pid, fid)
    o, _, _ = pooled_reference(van.astype(np.float64), H, gh, gw, FORCE_POOL[k], ks, pid, fid)
    assert list(ks) == [k]
    assert_pooled_close(g, o)


def test_van_pool_unaligned_layer_and_nan():
    """A layer of 45 values (the CV's scalar path) and a NaN VaN (its layer's
    CV is NaN: no pooling)."""
    gh, gw, f = 3, 3, 5
    van = _van_case(2, 1, gh, gw, f, (0.2, 0.2), seed=9)
    van[1, 7] = np.nan
    ipv.init(device=0, dtype="bf16", max_head_dim=64, max_frame_tokens=9, max_slabs=2,
             token_capacity=45, van_pool=True, cv_tau=(0.3, 0.9, 3.0))
    g, ks = _run_van_pool(van, 2, 1, gh, gw, (0.3, 0.9, 3.0))
    o, ko, _ = pooled_reference(van.astype(np.float64), 1, gh, gw, (0.3, 0.9, 3.0), ks)
    assert list(ks) == [7, 1] and list(ko) == [7, 1]
    assert_pooled_close(g, o)


# ------------------------------------------------------------ the whole pass
def _pool_workload(L=4, H=2, D=64, gh=7, gw=7, f=16, budget_frames=10, dtype="bf16", seed=3):
    return synth.CONFIGS["llava_pool"].scaled(n_layers=L, n_kv_heads=H, head_dim=D, grid_h=gh,
                                              grid_w=gw, n_frames=f, budget=budget_frames * gh * gw,
                                              dtype=dtype, seed=seed)


def check_pooled_pass(cache, w, N, tau, pid_valid):
    """One pooled pass on `cache` (live rows 0..N-1), checked end to end."""
    L, H, D, gh, gw, B = w.n_layers, w.n_kv_heads, w.head_dim, w.grid_h, w.grid_w, w.budget
    p, S = w.p, cache.n_slabs
    r = ipv.recent_frames(N // p)
    n_past = N - r * p
    cache.n_tokens = N
    k_src, v_src = to_np(cache.k_live), to_np(cache.v_live)
    pid_src = to_np(cache.pid_live) if pid_valid else None
    fid_src = cache.fid[cache.cur].cpu().numpy().view(np.uint32) if pid_valid else None
    k_s, v_s = cache.structs(pid_valid)
    tar_g = torch.empty((S, N), dtype=torch.float32, device="cuda")
    van_g = torch.empty_like(tar_g)
    ipv.score(k_s, v_s, L, H, D, N, gh, gw, tar_g, van_g)
    pooled_g = torch.empty_like(tar_g)
    ks_g = torch.empty((L,), dtype=torch.int32, device="cuda")
    ipv.van_pool(van_g, L, H, N, gh, gw, tau, pooled_g, ks_g,
                 None if not pid_valid else cache.pid[cache.cur],
                 None if not pid_valid else cache.fid[cache.cur], cache.capacity)
    kept = torch.full((S, B), -7, dtype=torch.int32, device="cuda")
    cur0 = cache.cur
    cache.compress(L, H, gh, gw, B, w.tar_ratio, kept, pid_valid=pid_valid)
    torch.cuda.synchronize()
    assert cache.cur != cur0
    kept_np, tg, vg = to_np(kept), to_np(tar_g), to_np(van_g)
    pg, ks = to_np(pooled_g), to_np(ks_g)
    # scores: TaR and VaN of past rows, VaN of the recent rows (the CV counts them)
    o_tar, o_van = oracle.scores(k_src, v_src, N, p, r, pid_src)
    assert_scores_close(tg, vg, o_tar, o_van, n_past)
    o_all = oracle.van_all(v_src, N)
    err = np.abs(vg[:, n_past:] - o_all[:, n_past:]) / o_all[:, n_past:]
    assert err.max() <= 1e-5
    # pooled VaN and pool sizes
    o_pool, ko, _ = pooled_reference(o_all, H, gh, gw, tau, ks,
                                     None if pid_src is None else pid_src[:, :N].copy(),
                                     None if fid_src is None else fid_src[:, :N].copy())
    assert_pooled_close(pg, o_pool, rows=n_past)
    # the pass against the whole oracle pass (same pool sizes) and against the rule
    n_diff = assert_selection_matches(kept_np, tg, pg, o_tar, o_pool, N, p, r, B, w.tar_ratio)
    assert_gather_exact(k_src, to_np(cache.k_live), kept_np, B)
    assert_gather_exact(v_src, to_np(cache.v_live), kept_np, B)
    pd = to_np(cache.pid_live)[:, :B]
    fd = cache.fid[cache.cur].cpu().numpy().view(np.uint32)[:, :B]
    want_p = np.take_along_axis(pid_src, kept_np, 1) if pid_src is not None else (kept_np % p)
    want_f = np.take_along_axis(fid_src, kept_np, 1) if fid_src is not None else (kept_np // p)
    assert np.array_equal(pd, want_p.astype(np.uint16)) and np.array_equal(fd, want_f.astype(np.uint32))
    if np.array_equal(ks, ko):
        o_kept = oracle.compress_pooled(k_src, v_src, N, gh, gw, r, B, float(np.float32(w.tar_ratio)), tau, H,
                                        None if pid_src is None else pid_src,
                                        None if fid_src is None else fid_src)[0]
        if n_diff == 0:
            assert np.array_equal(o_kept, kept_np)
    return ks, n_diff


def _pool_cache(w, cap):
    return PingPongCache(w.n_slabs, cap, w.head_dim, w.dtype, patch_ids=True, frame_ids=True)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_pooled_pass_fresh_then_compacted(dtype):
    """A fresh cache (ids derived), then the compacted half with 6 new frames
    appended (ids carried): two pooled passes against the oracle."""
    w = _pool_workload(dtype=dtype)
    p, N, B = w.p, w.n_tokens, w.budget
    K, V = synth.host_generate(w, n_frames=w.n_frames + 6)
    o_all = oracle.van_all(V[:, :N], N)
    tau = spread_tau(oracle.van_pool(o_all, w.n_kv_heads, w.grid_h, w.grid_w, (0, 0, 0))[2],
                     w.cv_tau)
    ipv.init(device=0, dtype=dtype, max_head_dim=w.head_dim, max_frame_tokens=p,
             max_slabs=w.n_slabs, token_capacity=N, van_pool=True, cv_tau=tau)
    cache = _pool_cache(w, N)
    cache.k.zero_()
    cache.v.zero_()
    cache.k[0] = to_dev(K[:, :N], dtype)
    cache.v[0] = to_dev(V[:, :N], dtype)
    ks1, _ = check_pooled_pass(cache, w, N, tau, pid_valid=False)
    assert len(set(ks1.tolist())) > 1
    # append frames f .. f+5 behind the B survivors: patch ids 0..p-1, fresh frame ids
    c = cache.cur
    cache.k[c, :, B:N] = to_dev(K[:, N:N + 6 * p], dtype)
    cache.v[c, :, B:N] = to_dev(V[:, N:N + 6 * p], dtype)
    cache.pid[c, :, B:N] = torch.arange(p, dtype=torch.int16, device="cuda").repeat(6)
    frames = torch.arange(w.n_frames, w.n_frames + 6, dtype=torch.int32, device="cuda")
    cache.fid[c, :, B:N] = frames.repeat_interleave(p)
    check_pooled_pass(cache, w, N, tau, pid_valid=True)


def test_pooled_pass_requires_frame_ids_with_patch_ids():
    w = _pool_workload()
    ipv.init(device=0, dtype="bf16", max_head_dim=w.head_dim, max_frame_tokens=w.p,
             max_slabs=w.n_slabs, token_capacity=w.n_tokens, van_pool=True, cv_tau=w.cv_tau)
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, "bf16", patch_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.pid.zero_()
    cache.n_tokens = w.n_tokens
    kept = torch.empty((w.n_slabs, w.budget), dtype=torch.int32, device="cuda")
    with pytest.raises(ipv.IpvError) as ei:
        cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, w.budget, 0.5, kept)
    assert ei.value.status == ipv.IPV_EINVAL and "frame ids" in str(ei.value)


def test_pooled_llava_full_size_sampled_layers():
    """The LLaVA-OV-7B pooled workload (28 x 4 slabs, 9408 -> 6272) as the
    bench runs it; the oracle checks four whole layers (the CV spans a
    layer's heads)."""
    w = synth.CONFIGS["llava_pool"]
    S, N, B, D, p = w.n_slabs, w.n_tokens, w.budget, w.head_dim, w.p
    ipv.init(device=0, dtype=w.dtype, max_head_dim=D, max_frame_tokens=p, max_slabs=S,
             token_capacity=N, van_pool=True, cv_tau=w.cv_tau)
    cache = _pool_cache(w, N)
    synth.device_generate(w, cache.k[0], cache.v[0])
    layers = [0, 9, 18, 27]
    sel = np.concatenate([np.arange(l * w.n_kv_heads, (l + 1) * w.n_kv_heads) for l in layers])
    sel_t = torch.as_tensor(sel, device="cuda")
    k_src = to_np(cache.k[0].index_select(0, sel_t))
    v_src = to_np(cache.v[0].index_select(0, sel_t))
    cache.n_tokens = N
    k_s, v_s = cache.structs(pid_valid=False)
    tar_g = torch.empty((S, N), dtype=torch.float32, device="cuda")
    van_g = torch.empty_like(tar_g)
    ipv.score(k_s, v_s, w.n_layers, w.n_kv_heads, D, N, w.grid_h, w.grid_w, tar_g, van_g)
    pooled_g = torch.empty_like(tar_g)
    ks_g = torch.empty((w.n_layers,), dtype=torch.int32, device="cuda")
    ipv.van_pool(van_g, w.n_layers, w.n_kv_heads, N, w.grid_h, w.grid_w, w.cv_tau, pooled_g, ks_g)
    kept = torch.empty((S, B), dtype=torch.int32, device="cuda")
    cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, B, w.tar_ratio, kept,
                   pid_valid=False)
    torch.cuda.synchronize()
    ks_all = to_np(ks_g)
    assert sorted(set(ks_all.tolist())) == [1, 3, 5, 7]
    r = ipv.recent_frames(w.n_frames)
    n_past = N - r * p
    tg = to_np(tar_g.index_select(0, sel_t))
    vg = to_np(van_g.index_select(0, sel_t))
    pg = to_np(pooled_g.index_select(0, sel_t))
    kept_np = to_np(kept.index_select(0, sel_t))
    o_tar, o_van = oracle.scores(k_src, v_src, N, p, r)
    assert_scores_close(tg, vg, o_tar, o_van, n_past)
    o_all = oracle.van_all(v_src, N)
    o_pool, _, _ = pooled_reference(o_all, w.n_kv_heads, w.grid_h, w.grid_w, w.cv_tau,
                                    ks_all[layers])
    assert_pooled_close(pg, o_pool, rows=n_past)
    assert_selection_matches(kept_np, tg, pg, o_tar, o_pool, N, p, r, B, w.tar_ratio)
    assert_gather_exact(k_src, to_np(cache.k_live.index_select(0, sel_t)), kept_np, B)
    assert_gather_exact(v_src, to_np(cache.v_live.index_select(0, sel_t)), kept_np, B)
    fd = cache.fid[cache.cur].index_select(0, sel_t).cpu().numpy()[:, :B]
    assert np.array_equal(fd, kept_np // p)


def test_raw_and_pooled_passes_differ_only_in_the_van_stage():
    """With every layer at pool size 1 the pooled pass equals the raw pass
    bit for bit (K, V, indices)."""
    w = _pool_workload()
    K, V = synth.host_generate(w)
    outs = []
    for pooled in (False, True):
        ipv.init(device=0, dtype=w.dtype, max_head_dim=w.head_dim, max_frame_tokens=w.p,
                 max_slabs=w.n_slabs, token_capacity=w.n_tokens, van_pool=pooled,
                 cv_tau=FORCE_POOL[1])
        cache = _pool_cache(w, w.n_tokens)
        cache.k[0] = to_dev(K, w.dtype)
        cache.v[0] = to_dev(V, w.dtype)
        cache.n_tokens = w.n_tokens
        kept = torch.empty((w.n_slabs, w.budget), dtype=torch.int32, device="cuda")
        cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, w.budget, w.tar_ratio, kept,
                       pid_valid=False)
        torch.cuda.synchronize()
        B = w.budget
        outs.append((to_np(kept), to_np(cache.k_live)[:, :B], to_np(cache.v_live)[:, :B]))
        ipv.shutdown()
    for a, b in zip(*outs):
        assert np.array_equal(a, b)
