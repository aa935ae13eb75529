"""GPU parity of the per-layer shared index set (Sec. 3.1: K in R^{H x N x D}
compressed as K[:, I, :], one I per layer) against the CPU oracle, through
the C ABI: per-layer scores, whole passes on fresh and compacted caches,
with and without pooled VaN, and the LLaVA shape on sampled layers.
Rules: parity.py.
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


def _init(w, cap, van_pool=False, cv_tau=(0.0, 0.0, 0.0), shared=True):
    ipv.init(device=0, dtype=w.dtype, max_head_dim=w.head_dim, max_frame_tokens=w.p,
             max_slabs=w.n_slabs, token_capacity=cap, van_pool=van_pool, cv_tau=cv_tau,
             head_shared=shared)


def _cache(w, cap, K, V):
    cache = PingPongCache(w.n_slabs, cap, w.head_dim, w.dtype, patch_ids=True, frame_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.k[0, :, :K.shape[1]] = to_dev(K, w.dtype)
    cache.v[0, :, :V.shape[1]] = to_dev(V, w.dtype)
    return cache


def check_shared_pass(cache, w, N, pid_valid, tau=None):
    """One shared-index pass (pooled VaN if tau) on live rows 0..N-1, checked."""
    L, H, D, gh, gw, B, p = w.n_layers, w.n_kv_heads, w.head_dim, w.grid_h, w.grid_w, w.budget, w.p
    r = ipv.recent_frames(N // p)
    n_past = N - r * p
    cache.n_tokens = N
    k_src, v_src = to_np(cache.k_live), to_np(cache.v_live)
    pid_src = to_np(cache.pid_live) if pid_valid else None
    fid_src = cache.fid[cache.cur].cpu().numpy().view(np.uint32) if pid_valid else None
    k_s, v_s = cache.structs(pid_valid)
    tar_g = torch.empty((L, N), dtype=torch.float32, device="cuda")
    van_g = torch.empty_like(tar_g)
    ipv.score(k_s, v_s, L, H, D, N, gh, gw, tar_g, van_g)
    sel_van = van_g
    ks = None
    if tau is not None:
        pooled_g = torch.empty_like(van_g)
        ks_g = torch.empty((L,), dtype=torch.int32, device="cuda")
        ipv.van_pool(van_g, L, 1, N, gh, gw, tau, pooled_g, ks_g,
                     cache.pid[cache.cur][::H] if pid_valid else None,
                     cache.fid[cache.cur][::H] if pid_valid else None, H * cache.capacity)
        sel_van = pooled_g
    kept = torch.full((L, B), -7, dtype=torch.int32, device="cuda")
    cur0 = cache.cur
    cache.compress(L, H, gh, gw, B, w.tar_ratio, kept, pid_valid=pid_valid)
    torch.cuda.synchronize()
    assert cache.cur != cur0
    kept_np, tg, vg = to_np(kept), to_np(tar_g), to_np(van_g)
    o_tar, o_van = oracle.scores_shared(k_src, v_src, H, N, p, r, pid_src)
    assert_scores_close(tg, vg, o_tar, o_van, n_past)
    assert np.all(tg[:, n_past:] == 0)
    if tau is None:
        assert np.all(vg[:, n_past:] == 0)
        g_sel, o_sel = vg, o_van
    else:
        o_all = oracle.van_all_shared(v_src, H, N)
        err = np.abs(vg[:, n_past:] - o_all[:, n_past:]) / o_all[:, n_past:]
        assert err.max() <= 1e-5
        ks = to_np(ks_g)
        o_sel, _, _ = pooled_reference(o_all, 1, gh, gw, tau, ks,
                                       None if pid_src is None else pid_src[::H, :N].copy(),
                                       None if fid_src is None else fid_src[::H, :N].copy())
        g_sel = to_np(sel_van)
        assert_pooled_close(g_sel, o_sel, rows=n_past)
    n_diff = assert_selection_matches(kept_np, tg, g_sel, o_tar, o_sel, N, p, r, B, w.tar_ratio)
    kept_slab = np.repeat(kept_np, H, axis=0)       # every head takes its layer's rows
    assert_gather_exact(k_src, to_np(cache.k_live), kept_slab, B)
    assert_gather_exact(v_src, to_np(cache.v_live), kept_slab, B)
    pd = to_np(cache.pid_live)[:, :B]
    fd = cache.fid[cache.cur].cpu().numpy().view(np.uint32)[:, :B]
    want_p = np.take_along_axis(pid_src, kept_slab, 1) if pid_src is not None else kept_slab % p
    want_f = np.take_along_axis(fid_src, kept_slab, 1) if fid_src is not None else kept_slab // p
    assert np.array_equal(pd, want_p.astype(np.uint16)) and np.array_equal(fd, want_f.astype(np.uint32))
    if n_diff == 0:
        o = oracle.compress_shared(k_src, v_src, N, gh, gw, r, B, float(np.float32(w.tar_ratio)), H,
                                   pid_src, fid_src,
                                   tau=tau)
        if tau is None or np.array_equal(o[5], ks):
            assert np.array_equal(o[0], kept_np)
    return n_diff


def _workload(dtype="bf16", H=4, D=128, gh=7, gw=7, f=16, budget_frames=10, L=3, **kw):
    base = synth.CONFIGS["llava_pool"] if kw.pop("pool", False) else synth.CONFIGS["llava"]
    return base.scaled(n_layers=L, n_kv_heads=H, head_dim=D, grid_h=gh, grid_w=gw, n_frames=f,
                       budget=budget_frames * gh * gw, dtype=dtype, **kw)


@pytest.mark.parametrize("dtype,H,D", [("bf16", 4, 128), ("f32", 2, 64), ("bf16", 8, 128),
                                       ("f32", 3, 32)])
def test_shared_pass_fresh_then_compacted(dtype, H, D):
    w = _workload(dtype=dtype, H=H, D=D, seed=H)
    p, N, B = w.p, w.n_tokens, w.budget
    K, V = synth.host_generate(w, n_frames=w.n_frames + 6)
    _init(w, N)
    cache = _cache(w, N, K[:, :N], V[:, :N])
    check_shared_pass(cache, w, N, pid_valid=False)
    c = cache.cur
    cache.k[c, :, B:N] = to_dev(K[:, N:N + 6 * p], dtype)
    cache.v[c, :, B:N] = to_dev(V[:, N:N + 6 * p], dtype)
    cache.pid[c, :, B:N] = torch.arange(p, dtype=torch.int16, device="cuda").repeat(6)
    cache.fid[c, :, B:N] = torch.arange(w.n_frames, w.n_frames + 6, dtype=torch.int32,
                                        device="cuda").repeat_interleave(p)
    check_shared_pass(cache, w, N, pid_valid=True)


def test_shared_pooled_pass_fresh_then_compacted():
    w = _workload(pool=True, L=4, seed=11)
    p, N, B = w.p, w.n_tokens, w.budget
    K, V = synth.host_generate(w, n_frames=w.n_frames + 6)
    cv = oracle.van_pool(oracle.van_all_shared(V[:, :N], w.n_kv_heads, N), 1, w.grid_h, w.grid_w,
                         (0, 0, 0))[2]
    c_sorted = np.sort(cv)
    tau = tuple(float(np.float32(0.5 * (c_sorted[i] + c_sorted[i + 1]))) for i in range(3))
    _init(w, N, van_pool=True, cv_tau=tau)
    cache = _cache(w, N, K[:, :N], V[:, :N])
    check_shared_pass(cache, w, N, pid_valid=False, tau=tau)
    c = cache.cur
    cache.k[c, :, B:N] = to_dev(K[:, N:N + 6 * p], w.dtype)
    cache.v[c, :, B:N] = to_dev(V[:, N:N + 6 * p], w.dtype)
    cache.pid[c, :, B:N] = torch.arange(p, dtype=torch.int16, device="cuda").repeat(6)
    cache.fid[c, :, B:N] = torch.arange(w.n_frames, w.n_frames + 6, dtype=torch.int32,
                                        device="cuda").repeat_interleave(p)
    check_shared_pass(cache, w, N, pid_valid=True, tau=tau)


def test_one_head_shared_equals_per_head():
    """With one KV head the shared index set is the per-head pass: bit for bit."""
    w = _workload(H=1, L=6, seed=2)
    K, V = synth.host_generate(w)
    outs = []
    for shared in (False, True):
        _init(w, w.n_tokens, shared=shared)
        cache = _cache(w, w.n_tokens, K, V)
        cache.n_tokens = w.n_tokens
        kept = torch.empty((w.n_slabs, w.budget), dtype=torch.int32, device="cuda")
        cache.compress(w.n_layers, 1, w.grid_h, w.grid_w, w.budget, w.tar_ratio, kept, pid_valid=False)
        k_s, v_s = cache.structs(pid_valid=False)
        torch.cuda.synchronize()
        outs.append((to_np(kept), to_np(cache.k_live)[:, :w.budget], to_np(cache.v_live)[:, :w.budget]))
        ipv.shutdown()
    for a, b in zip(*outs):
        assert np.array_equal(a, b)


def test_shared_llava_full_size_sampled_layers():
    w = synth.CONFIGS["llava"]
    S, N, B, D, p, H = w.n_slabs, w.n_tokens, w.budget, w.head_dim, w.p, w.n_kv_heads
    _init(w, N)
    cache = PingPongCache(S, N, D, w.dtype, patch_ids=True, frame_ids=True)
    synth.device_generate(w, cache.k[0], cache.v[0])
    layers = np.array([0, 13, 27])
    sel = np.concatenate([np.arange(l * H, (l + 1) * H) for l in layers])
    sel_t = torch.as_tensor(sel, device="cuda")
    k_src = to_np(cache.k[0].index_select(0, sel_t))
    v_src = to_np(cache.v[0].index_select(0, sel_t))
    cache.n_tokens = N
    k_s, v_s = cache.structs(pid_valid=False)
    tar_g = torch.empty((w.n_layers, N), dtype=torch.float32, device="cuda")
    van_g = torch.empty_like(tar_g)
    ipv.score(k_s, v_s, w.n_layers, H, D, N, w.grid_h, w.grid_w, tar_g, van_g)
    kept = torch.empty((w.n_layers, B), dtype=torch.int32, device="cuda")
    cache.compress(w.n_layers, H, w.grid_h, w.grid_w, B, w.tar_ratio, kept, pid_valid=False)
    torch.cuda.synchronize()
    r = ipv.recent_frames(w.n_frames)
    lt = torch.as_tensor(layers, device="cuda")
    tg, vg = to_np(tar_g.index_select(0, lt)), to_np(van_g.index_select(0, lt))
    kept_np = to_np(kept.index_select(0, lt))
    o_tar, o_van = oracle.scores_shared(k_src, v_src, H, N, p, r)
    assert_scores_close(tg, vg, o_tar, o_van, N - r * p)
    assert_selection_matches(kept_np, tg, vg, o_tar, o_van, N, p, r, B, w.tar_ratio)
    kept_slab = np.repeat(kept_np, H, axis=0)
    assert_gather_exact(k_src, to_np(cache.k_live.index_select(0, sel_t)), kept_slab, B)
    assert_gather_exact(v_src, to_np(cache.v_live.index_select(0, sel_t)), kept_slab, B)


def test_shared_rejects_wide_blocks_and_single_kernel():
    w = _workload(H=16, D=128, L=1)                 # 16 x 128 bf16 = 4 KB per token block
    _init(w, w.n_tokens)
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype, patch_ids=False)
    cache.k.zero_()
    cache.v.zero_()
    cache.n_tokens = w.n_tokens
    kept = torch.empty((1, w.budget), dtype=torch.int32, device="cuda")
    with pytest.raises(ipv.IpvError) as ei:
        cache.compress(1, 16, w.grid_h, w.grid_w, w.budget, 0.5, kept, pid_valid=False)
    assert ei.value.status == ipv.IPV_EINVAL and "2048" in str(ei.value)
    ipv.shutdown()
    with pytest.raises(ipv.IpvError):
        ipv.init(device=0, dtype="bf16", max_head_dim=128, max_frame_tokens=49, max_slabs=4,
                 token_capacity=784, single_kernel=True, head_shared=True)
