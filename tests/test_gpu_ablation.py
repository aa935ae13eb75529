"""GPU parity of the ablation variants (Sec. 4 ablation table: TaR Reverse,
VaN Reverse, TaR Frame, Uniform Select) against the CPU oracle, through the
C ABI, on a fresh cache and on its compacted half with new frames appended
(patch and frame ids). Rules: parity.py, applied to the scores each variant
ranks; Uniform Select reads no score, so its indices are checked bit for
bit."""
import numpy as np
import pytest

import oracle
import synth
from parity import assert_gather_exact, assert_selection_matches

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


def check_ablation_pass(cache, w, N, variant, pid_valid):
    """One pass of a score-ranking variant on live rows 0..N-1, checked against
    the oracle on the scores that variant ranks."""
    L, H, D, gh, gw, B, p = w.n_layers, w.n_kv_heads, w.head_dim, w.grid_h, w.grid_w, w.budget, w.p
    r = ipv.recent_frames(N // p)
    n_past = N - r * p
    cache.n_tokens = N
    S = cache.n_slabs
    k_src, v_src = to_np(cache.k_live), to_np(cache.v_live)
    pid_src = to_np(cache.pid_live) if pid_valid else None
    fid_src = cache.fid[cache.cur].cpu().numpy().view(np.uint32) if pid_valid else None
    k_s, v_s = cache.structs(pid_valid)
    tar_g = torch.empty((S, N), dtype=torch.float32, device="cuda")
    van_g = torch.empty_like(tar_g)
    ipv.score(k_s, v_s, L, H, D, N, gh, gw, tar_g, van_g)
    kept = torch.full((S, B), -7, dtype=torch.int32, device="cuda")
    cache.compress(L, H, gh, gw, B, w.tar_ratio, kept, pid_valid=pid_valid)
    torch.cuda.synchronize()
    kept_np = to_np(kept)
    tg = to_np(tar_g).astype(np.float64)
    vg = to_np(van_g).astype(np.float64)
    o_tar, o_van = oracle.scores(k_src, v_src, N, p, r, pid_src)
    if variant == "tar_frame":
        o_tar = oracle.frame_mean(o_tar, n_past, p, fid_src)
    err = np.abs(tg[:, :n_past] - o_tar[:, :n_past]) / np.maximum(np.abs(o_tar[:, :n_past]), 1.0)
    assert err.max() <= 1e-5
    # the scores each stage ranks (a reversed stage ranks its negated scores)
    sgn_t = -1.0 if variant == "tar_reverse" else 1.0
    sgn_v = -1.0 if variant == "van_reverse" else 1.0
    n_diff = assert_selection_matches(kept_np, sgn_t * tg, sgn_v * vg, sgn_t * o_tar, sgn_v * o_van,
                                      N, p, r, B, w.tar_ratio)
    assert_gather_exact(k_src, to_np(cache.k_live), kept_np, B)
    assert_gather_exact(v_src, to_np(cache.v_live), kept_np, B)
    if n_diff == 0:
        o = oracle.compress_ablation(k_src, v_src, N, gh, gw, r, B, float(np.float32(w.tar_ratio)), variant,
                                     pid_src, fid_src)
        assert np.array_equal(o[0], kept_np)
    return n_diff


@pytest.mark.parametrize("variant", ["tar_reverse", "van_reverse", "tar_frame"])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_ablation_fresh_then_compacted(variant, dtype):
    w = synth.CONFIGS["llava"].scaled(n_layers=3, n_kv_heads=2, head_dim=64, grid_h=7, grid_w=7,
                                      n_frames=16, budget=10 * 49, dtype=dtype, seed=31)
    p, N, B = w.p, w.n_tokens, w.budget
    K, V = synth.host_generate(w, n_frames=w.n_frames + 6)
    ipv.init(device=0, dtype=dtype, max_head_dim=w.head_dim, max_frame_tokens=p,
             max_slabs=w.n_slabs, token_capacity=N, ablation=variant)
    cache = PingPongCache(w.n_slabs, N, w.head_dim, dtype, patch_ids=True, frame_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.k[0] = to_dev(K[:, :N], dtype)
    cache.v[0] = to_dev(V[:, :N], dtype)
    check_ablation_pass(cache, w, N, variant, pid_valid=False)
    c = cache.cur
    k, v = cache.structs(pid_valid=True)
    ipv.append_frames(k, v, to_dev(K[:, N:N + 6 * p], dtype), to_dev(V[:, N:N + 6 * p], dtype),
                      w.n_layers, w.n_kv_heads, w.head_dim, B, 6, w.grid_h, w.grid_w)
    check_ablation_pass(cache, w, N, variant, pid_valid=True)


def test_tar_frame_needs_frame_ids_with_patch_ids():
    w = synth.CONFIGS["tiny"]
    ipv.init(device=0, dtype=w.dtype, max_head_dim=w.head_dim, max_frame_tokens=w.p,
             max_slabs=w.n_slabs, token_capacity=w.n_tokens, ablation="tar_frame")
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype, patch_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.pid.zero_()
    cache.n_tokens = w.n_tokens
    kept = torch.empty((w.n_slabs, w.budget), dtype=torch.int32, device="cuda")
    with pytest.raises(ipv.IpvError) as ei:
        cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, w.budget, 0.5, kept)
    assert ei.value.status == ipv.IPV_EINVAL


def check_uniform_pass(cache, w, N, pid_valid, n_units):
    """One Uniform Select pass on live rows 0..N-1: indices equal the oracle's
    bit for bit (n_units rows: slabs, or layers with a shared index set, every
    head compacted with its unit's rows), bytes and ids exact."""
    B, p = w.budget, w.p
    H = w.n_slabs // n_units
    cache.n_tokens = N
    k_src, v_src = to_np(cache.k_live), to_np(cache.v_live)
    pid_src = to_np(cache.pid_live) if pid_valid else None
    fid_src = cache.fid[cache.cur].cpu().numpy().view(np.uint32) if pid_valid else None
    kept = torch.full((n_units, B), -7, dtype=torch.int32, device="cuda")
    cur0 = cache.cur
    cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, B, w.tar_ratio, kept,
                   pid_valid=pid_valid)
    sel = torch.full((n_units, B), -7, dtype=torch.int32, device="cuda")
    dummy = torch.zeros((n_units, N), dtype=torch.float32, device="cuda")
    ipv.select(dummy, dummy, n_units, N, w.grid_h, w.grid_w, B, w.tar_ratio, sel)
    torch.cuda.synchronize()
    assert cache.cur != cur0
    kept_np = to_np(kept)
    want = oracle.uniform_select(n_units, N, p, B)
    assert np.array_equal(kept_np, want)
    assert np.array_equal(to_np(sel), want)                        # ipv_select == the pass
    kept_slab = np.repeat(kept_np, H, axis=0)
    assert_gather_exact(k_src, to_np(cache.k_live), kept_slab, B)
    assert_gather_exact(v_src, to_np(cache.v_live), kept_slab, B)
    pd = to_np(cache.pid_live)[:, :B]
    fd = cache.fid[cache.cur].cpu().numpy().view(np.uint32)[:, :B]
    want_p = np.take_along_axis(pid_src, kept_slab, 1) if pid_src is not None else kept_slab % p
    want_f = np.take_along_axis(fid_src, kept_slab, 1) if fid_src is not None else kept_slab // p
    assert np.array_equal(pd, want_p.astype(np.uint16)) and np.array_equal(fd, want_f.astype(np.uint32))
    if H == 1:
        o = oracle.compress_ablation(k_src, v_src, N, w.grid_h, w.grid_w, ipv.recent_frames(N // p),
                                     B, w.tar_ratio, "uniform", pid_src, fid_src)
        assert np.array_equal(o[0], kept_np)


@pytest.mark.parametrize("dtype,shared", [("bf16", False), ("f32", False), ("bf16", True)])
def test_uniform_select_fresh_then_compacted(dtype, shared):
    """A fresh cache, then twice the compacted half with whole frames appended
    by ipv_append_frames: every cached frame stays whole, so each pass keeps
    whole frames at regular intervals of the frame view."""
    w = synth.CONFIGS["llava"].scaled(n_layers=3, n_kv_heads=2, head_dim=64, grid_h=5, grid_w=7,
                                      n_frames=17, budget=11 * 35, dtype=dtype, seed=41,
                                      head_shared=shared)
    p, N, B = w.p, w.n_tokens, w.budget
    n_new = (N - B) // p
    K, V = synth.host_generate(w, n_frames=w.n_frames + 2 * n_new)
    ipv.init(device=0, dtype=dtype, max_head_dim=w.head_dim, max_frame_tokens=p,
             max_slabs=w.n_slabs, token_capacity=N, ablation="uniform", head_shared=shared)
    cache = PingPongCache(w.n_slabs, N, w.head_dim, dtype, patch_ids=True, frame_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.k[0] = to_dev(K[:, :N], dtype)
    cache.v[0] = to_dev(V[:, :N], dtype)
    n_units = w.n_layers if shared else w.n_slabs
    check_uniform_pass(cache, w, N, False, n_units)
    for step in range(2):
        k, v = cache.structs(pid_valid=True)
        rows = slice(N + step * n_new * p, N + (step + 1) * n_new * p)
        ipv.append_frames(k, v, to_dev(K[:, rows], dtype), to_dev(V[:, rows], dtype), w.n_layers,
                          w.n_kv_heads, w.head_dim, B, n_new, w.grid_h, w.grid_w)
        check_uniform_pass(cache, w, N, True, n_units)


def test_uniform_select_needs_whole_frames():
    w = synth.CONFIGS["tiny"]
    ipv.init(device=0, dtype=w.dtype, max_head_dim=w.head_dim, max_frame_tokens=w.p,
             max_slabs=w.n_slabs, token_capacity=w.n_tokens, ablation="uniform")
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype, patch_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.n_tokens = w.n_tokens
    kept = torch.empty((w.n_slabs, w.budget + 1), dtype=torch.int32, device="cuda")
    with pytest.raises(ipv.IpvError) as ei:
        cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, w.budget + 1, 0.5, kept,
                       pid_valid=False)
    assert ei.value.status == ipv.IPV_EINVAL
    # a budget below the recent frames is accepted: Uniform Select has no recent-frame rule
    kept = torch.empty((w.n_slabs, w.p), dtype=torch.int32, device="cuda")
    cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, w.p, 0.5, kept, pid_valid=False)
    torch.cuda.synchronize()
    assert np.array_equal(to_np(kept), oracle.uniform_select(w.n_slabs, w.n_tokens, w.p, w.p))
