"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Inputs are seeded synthetic caches (synth/); both sides read the same bytes.
Scores, indices and compacted bytes are checked with the rules in parity.py.
"""
import numpy as np
import pytest

import oracle
import synth
from parity import assert_gather_exact, assert_scores_close, assert_selection_matches

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


def init_for(S, cap, D, p, dtype, recent_frames=0, single_kernel=False):
    ipv.init(device=0, dtype=dtype, recent_frames=recent_frames, max_head_dim=D,
             max_frame_tokens=p, max_slabs=S, token_capacity=cap, single_kernel=single_kernel)


def check_pass(cache, L, H, N, gh, gw, budget, alpha, pid_valid, slabs=None):
    """One compress pass on `cache` (live rows 0..N-1) checked end to end.
    slabs: optional subset of slab indices for the oracle (large cases)."""
    p = gh * gw
    S, D = cache.n_slabs, cache.head_dim
    r = ipv.recent_frames(N // p)
    sel = np.arange(S) if slabs is None else np.asarray(slabs)
    sel_t = torch.as_tensor(sel, device="cuda")
    cache.n_tokens = N
    k_src = to_np(cache.k_live.index_select(0, sel_t))
    v_src = to_np(cache.v_live.index_select(0, sel_t))
    pid_src = (to_np(cache.pid_live.index_select(0, sel_t))
               if (pid_valid and cache.pid is not None) else None)
    fid_src = (cache.fid[cache.cur].index_select(0, sel_t).cpu().numpy()
               if (pid_valid and cache.fid is not None) else None)
    k_struct, v_struct = cache.structs(pid_valid)
    tar_g = torch.empty((S, N), dtype=torch.float32, device="cuda")
    van_g = torch.empty_like(tar_g)
    has_past = r * p < N
    if has_past:
        ipv.score(k_struct, v_struct, L, H, D, N, gh, gw, tar_g, van_g)
    kept_sel = torch.empty((S, budget), dtype=torch.int32, device="cuda")
    if has_past:
        ipv.select(tar_g, van_g, S, N, gh, gw, budget, alpha, kept_sel)
    kept = torch.full((S, budget), -7, dtype=torch.int32, device="cuda")
    cur_before = cache.cur
    cache.compress(L, H, gh, gw, budget, alpha, kept, pid_valid=pid_valid)
    torch.cuda.synchronize()
    kept_np = to_np(kept.index_select(0, sel_t))
    if N <= budget:  # pass-through
        assert cache.cur == cur_before
        want = np.array(list(range(N)) + [-1] * (budget - N), np.int32)
        assert np.all(kept_np == want)
        return None
    assert cache.cur != cur_before
    assert np.array_equal(to_np(kept_sel.index_select(0, sel_t)), kept_np)  # ipv_select == the pass
    o_tar, o_van = oracle.scores(k_src, v_src, N, p, r, pid_src)
    tg, vg = to_np(tar_g.index_select(0, sel_t)), to_np(van_g.index_select(0, sel_t))
    errs = assert_scores_close(tg, vg, o_tar, o_van, N - r * p)
    assert np.all(tg[:, N - r * p:] == 0) and np.all(vg[:, N - r * p:] == 0)
    n_diff = assert_selection_matches(kept_np, tg, vg, o_tar, o_van, N, p, r, budget, alpha)
    assert_gather_exact(k_src, to_np(cache.k_live.index_select(0, sel_t)), kept_np, budget)
    assert_gather_exact(v_src, to_np(cache.v_live.index_select(0, sel_t)), kept_np, budget)
    if cache.pid is not None:
        pd = to_np(cache.pid_live.index_select(0, sel_t))[:, :budget]
        want = (np.take_along_axis(pid_src, kept_np, 1) if pid_src is not None
                else (kept_np % p).astype(np.uint16))
        assert np.array_equal(pd, want)
    if cache.fid is not None:  # frame ids travel with their rows too
        fd = cache.fid[cache.cur].index_select(0, sel_t).cpu().numpy()[:, :budget]
        want = (np.take_along_axis(fid_src, kept_np, 1) if fid_src is not None
                else (kept_np // p).astype(np.int32))
        assert np.array_equal(fd, want)
    return errs, n_diff


def host_case(S, f, gh, gw, D, dtype, seed, static_frac=0.7, cap_extra=0):
    w = synth.Workload("case", 1, S, D, dtype, gh, gw, f, 1, 0.5, static_frac=static_frac, seed=seed)
    K, V = synth.host_generate(w)
    cap = f * gh * gw + cap_extra
    cache = PingPongCache(S, cap, D, dtype, patch_ids=True)
    cache.k.zero_()
    cache.v.zero_()
    cache.k[0, :, :f * gh * gw] = to_dev(K, dtype)
    cache.v[0, :, :f * gh * gw] = to_dev(V, dtype)
    return cache


def test_tiny_config():
    """1 layer x 2 heads, D=64 fp32, 8 frames of 4x4, budget 48, alpha 0.5, seed 0."""
    w = synth.CONFIGS["tiny"]
    init_for(w.n_slabs, w.n_tokens, w.head_dim, w.p, w.dtype)
    K, V = synth.host_generate(w)
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype)
    cache.k[0] = to_dev(K, w.dtype)
    cache.v[0] = to_dev(V, w.dtype)
    errs, n_diff = check_pass(cache, w.n_layers, w.n_kv_heads, w.n_tokens, w.grid_h, w.grid_w,
                              w.budget, w.tar_ratio, pid_valid=False)
    assert n_diff == 0
    # The compacted half (with its patch ids) is a valid input for the next pass.
    cache2 = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype)
    cache2.k[0] = to_dev(K, w.dtype)
    cache2.v[0] = to_dev(V, w.dtype)
    cache2.pid[0] = torch.arange(w.n_tokens, device="cuda").remainder(w.p).to(torch.int16)
    check_pass(cache2, w.n_layers, w.n_kv_heads, w.n_tokens, w.grid_h, w.grid_w, w.budget,
               w.tar_ratio, pid_valid=True)
    B = w.budget
    assert torch.equal(cache2.k[1, :, :B], cache.k[1, :, :B])
    assert torch.equal(cache2.pid[1, :, :B], cache.pid[1, :, :B])


EDGE_CASES = [
    # S, f, gh, gw, D, dtype, budget_fn(N, p, rp), alpha
    (3, 12, 14, 14, 128, "bf16", lambda N, p, rp: N // 2 + 37, 0.5),      # ragged budget, many tiles
    (5, 40, 1, 7, 64, "bf16", lambda N, p, rp: 150, 0.3),                 # half-warp lanes idle
    (2, 16, 4, 4, 96, "bf16", lambda N, p, rp: rp + 1, 0.5),              # minimal budget
    (3, 20, 2, 5, 128, "f32", lambda N, p, rp: N - 1, 0.7),               # evict one token
    (4, 30, 1, 3, 32, "f32", lambda N, p, rp: 40, 0.0),                   # VaN only
    (2, 16, 7, 7, 256, "bf16", lambda N, p, rp: 400, 1.0),                # TaR only, 2 chunks/lane
    (2, 10, 3, 3, 512, "bf16", lambda N, p, rp: 50, 0.5),                 # 4 chunks/lane
    (2, 10, 3, 3, 512, "f32", lambda N, p, rp: 50, 0.5),                  # 8 chunks/lane
    (1, 9, 1, 1, 64, "bf16", lambda N, p, rp: 4, 0.5),                    # p = 1
    (2, 8, 4, 4, 64, "f32", lambda N, p, rp: N, 0.5),                     # pass-through N == C
    (2, 8, 4, 4, 64, "f32", lambda N, p, rp: N + 9, 0.5),                 # pass-through N < C
    (2, 9, 20, 20, 128, "bf16", lambda N, p, rp: 5 * p + 17, 0.5),        # m table > 200 KB: read via L2
    (1, 8, 9, 12, 512, "f32", lambda N, p, rp: 3 * p, 0.7),              # the same at 2 KB rows
]


@pytest.mark.parametrize("case", range(len(EDGE_CASES)))
def test_edge_shapes(case):
    S, f, gh, gw, D, dtype, budget_fn, alpha = EDGE_CASES[case]
    p = gh * gw
    N = f * p
    cap = N + 64
    budget = budget_fn(N, p, oracle.recent_frames(f) * p)
    assert budget <= cap
    init_for(S, cap, D, p, dtype)
    cache = host_case(S, f, gh, gw, D, dtype, seed=100 + case, cap_extra=64)
    check_pass(cache, 1, S, N, gh, gw, budget, alpha, pid_valid=False)


@pytest.mark.parametrize("r", [1, 3])
def test_recent_frames_override(r):
    S, f, gh, gw, D = 3, 10, 4, 5, 128
    init_for(S, f * gh * gw, D, gh * gw, "bf16", recent_frames=r)
    assert ipv.recent_frames(f) == r
    cache = host_case(S, f, gh, gw, D, "bf16", seed=7)
    check_pass(cache, 1, S, f * gh * gw, gh, gw, 90, 0.5, pid_valid=False)


def test_patch_ids_are_followed():
    """Past rows shuffled together with their patch ids score as before."""
    S, f, gh, gw, D = 2, 12, 3, 4, 128
    p, N = gh * gw, f * gh * gw
    init_for(S, N, D, p, "bf16")
    cache = host_case(S, f, gh, gw, D, "bf16", seed=11)
    r = ipv.recent_frames(f)
    n_past = N - r * p
    perm = torch.from_numpy(np.random.default_rng(3).permutation(n_past)).cuda()
    cache.k[0, :, :n_past] = cache.k[0, :, perm].clone()
    cache.v[0, :, :n_past] = cache.v[0, :, perm].clone()
    pid = torch.arange(N, device="cuda").remainder(p)
    pid[:n_past] = perm.remainder(p)
    cache.pid[0] = pid.to(torch.int16).expand(S, N)
    check_pass(cache, 1, S, N, gh, gw, N // 2, 0.5, pid_valid=True)


def test_select_exact_on_ties_nan_and_signed_zero():
    """Step (iii) alone on crafted fp32 scores: bit-exact against the oracle."""
    rng = np.random.default_rng(5)
    S, f, p = 6, 20, 7
    N = f * p
    init_for(S, N, 64, p, "f32")
    tar = (rng.integers(-3, 3, size=(S, N)) / 2).astype(np.float32)   # heavy ties
    van = rng.integers(0, 4, size=(S, N)).astype(np.float32)
    tar[0, :50] = -1.0                    # all equal
    tar[1, ::3] = np.nan                  # NaN ranks lowest
    van[2, ::4] = np.nan
    tar[3, ::2] = -0.0                    # -0 and +0 tie, broken by index
    tar[3, 1::2] = 0.0
    van[4] = 2.5                          # all VaN equal
    for budget, alpha in [(60, 0.5), (30, 0.9), (139, 0.5), (25, 0.0), (70, 1.0)]:
        r = oracle.recent_frames(f)
        kept = torch.empty((S, budget), dtype=torch.int32, device="cuda")
        ipv.select(torch.from_numpy(tar).cuda(), torch.from_numpy(van).cuda(), S, N, 1, p,
                   budget, alpha, kept)
        want = oracle.select(tar.astype(np.float64), van.astype(np.float64), N, p, r, budget,
                             float(np.float32(alpha)))
        assert np.array_equal(to_np(kept), want), (budget, alpha)


def test_select_exact_when_boundary_bins_overflow():
    """Step (iii) on crafted scores whose boundary bin holds thousands of
    close, distinct values (and ties): the selection's exact search over key
    windows, bit-exact against the oracle."""
    rng = np.random.default_rng(8)
    S, f, p = 3, 64, 256
    N = f * p
    r = oracle.recent_frames(f)
    n_past = N - r * p
    init_for(S, N, 64, p, "f32")
    tar = rng.uniform(-1.0, 0.2, size=(S, N)).astype(np.float32)
    van = rng.uniform(0.0, 0.9, size=(S, N)).astype(np.float32)
    # slab 0: 4000 TaR values within 1e-4 (one bin of the [-1, 1] map), 500 above
    idx = rng.permutation(n_past)
    tar[0, idx[:4000]] = (0.3 + rng.integers(0, 3000, 4000) * 3e-8).astype(np.float32)
    tar[0, idx[4000:4500]] = rng.uniform(0.5, 1.0, 500).astype(np.float32)
    # slab 1: VaN of 6000 tokens within 1e-3 of 1, 1000 spread above, one at 1000
    tar[1, :2000] = 0.9  # TaR takes these (ties broken by index)
    van[1, :2000] = 0.1
    idx = 2000 + rng.permutation(n_past - 2000)
    van[1, idx[:6000]] = (1.0 + rng.integers(0, 8000, 6000) * 1.25e-7).astype(np.float32)
    van[1, idx[6000:7000]] = rng.uniform(10.0, 100.0, 1000).astype(np.float32)
    van[1, idx[7000]] = 1000.0
    # slab 2: both, with NaN and signed zeros in the clusters
    tar[2] = tar[0]
    van[2] = van[1]
    tar[2, idx[:200]] = np.nan
    van[2, idx[200:400]] = -0.0
    for budget, alpha in [(8096, 0.5), (12288, 0.3), (6000, 0.6)]:
        kept = torch.empty((S, budget), dtype=torch.int32, device="cuda")
        ipv.select(torch.from_numpy(tar).cuda(), torch.from_numpy(van).cuda(), S, N, 1, p,
                   budget, alpha, kept)
        want = oracle.select(tar.astype(np.float64), van.astype(np.float64), N, p, r, budget,
                             float(np.float32(alpha)))
        assert np.array_equal(to_np(kept), want), (budget, alpha)


def _extreme_scores(rng, S, N):
    """fp32 TaR / VaN rows with infinities, NaN, signed zeros, denormals,
    values far outside TaR's [-1, 1], VaN ranges far wider than 2048 and
    values on or next to the selection's bin edges."""
    f32 = np.float32
    tar = rng.uniform(-1.0, 1.0, size=(S, N)).astype(f32)
    van = rng.uniform(0.0, 3.0, size=(S, N)).astype(f32)
    # 0: VaN log-uniform over 60 decades (bins of width 2^89)
    van[0] = (10.0 ** rng.uniform(-30, 30, N)).astype(f32)
    # 1: VaN with +inf and -inf among finite values (no finite range)
    van[1, ::7] = np.inf
    van[1, 3::11] = -np.inf
    # 2: TaR far outside [-1, 1], with infinities and NaN
    tar[2] = rng.uniform(-3.0, 3.0, N).astype(f32)
    tar[2, ::13] = np.inf
    tar[2, 5::17] = -np.inf
    tar[2, 2::19] = np.nan
    # 3: denormals and signed zeros
    tar[3] = (rng.integers(-50, 50, N) * f32(1e-44)).astype(f32)
    van[3] = (rng.integers(0, 50, N) * f32(1e-44)).astype(f32)
    tar[3, ::5] = -0.0
    van[3, 1::5] = -0.0
    # 4: negative VaN over a wide range (as the Reverse ablation feeds it)
    van[4] = rng.uniform(-1e6, 1e6, N).astype(f32)
    # 5: values on TaR's bin edges (b - 1024) / 1024 and one ulp either side
    e = ((rng.integers(0, 2048, N) - 1024) / 1024.0).astype(f32)
    step = rng.integers(-1, 2, N)
    tar[5] = np.where(step < 0, np.nextafter(e, f32(-2)), np.where(step > 0, np.nextafter(e, f32(2)), e))
    van[5] = (rng.integers(0, 3000, N) / 3.0).astype(f32)
    # 6: every VaN the same huge value, every TaR -inf
    van[6] = f32(1e30)
    tar[6] = -np.inf
    return tar, van


@pytest.mark.parametrize("f", [48, 200, 300])
def test_select_exact_on_extreme_scores(f):
    """Step (iii) alone on extreme fp32 scores, at slab sizes that take each
    selection kernel (scores in registers with 10 and 16 rows, keys in
    shared memory): bit-exact against the oracle's rule."""
    rng = np.random.default_rng(100 + f)
    S, p = 7, 64
    N = f * p
    r = oracle.recent_frames(f)
    init_for(S, N, 64, p, "f32")
    tar, van = _extreme_scores(rng, S, N)
    for frac, alpha in [(0.5, 0.5), (0.3, 0.9), (0.8, 0.2), (0.65, 1.0), (0.4, 0.0)]:
        budget = max(r * p + 1, int(frac * N))
        kept = torch.empty((S, budget), dtype=torch.int32, device="cuda")
        ipv.select(torch.from_numpy(tar).cuda(), torch.from_numpy(van).cuda(), S, N, 1, p,
                   budget, alpha, kept)
        want = oracle.select(tar.astype(np.float64), van.astype(np.float64), N, p, r, budget,
                             float(np.float32(alpha)))
        assert np.array_equal(to_np(kept), want), (f, budget, alpha)


@pytest.mark.parametrize("f", [1170, 1171, 10533, 10534, 18725, 18726, 32768, 32769])
def test_select_exact_at_kernel_size_limits(f):
    """One-token frames, so that the past tokens number exactly 1024 / 1025,
    9216 / 9217 and 16384 / 16385 (the last size each selection kernel takes,
    every row of every thread full, and the first one of the next), and
    28672 / 28673 (the keys-in-shared-memory kernel at the large config's
    size).
    Tied, NaN and signed-zero scores; bit-exact against the oracle."""
    rng = np.random.default_rng(f)
    S, p, N = 4, 1, f
    r = oracle.recent_frames(f)
    init_for(S, N, 64, p, "f32")
    tar = (rng.integers(-40, 40, size=(S, N)) / 40).astype(np.float32)
    van = rng.uniform(0.0, 2.0, size=(S, N)).astype(np.float32)
    van[:, ::3] = np.round(van[:, ::3], 1)
    tar[1, ::9] = np.nan
    van[2, 1::7] = np.nan
    tar[3, ::2] = -0.0
    for frac, alpha in [(0.5, 0.5), (0.9, 0.3)]:
        budget = max(r * p + 1, int(frac * N))
        kept = torch.empty((S, budget), dtype=torch.int32, device="cuda")
        ipv.select(torch.from_numpy(tar).cuda(), torch.from_numpy(van).cuda(), S, N, 1, 1,
                   budget, alpha, kept)
        want = oracle.select(tar.astype(np.float64), van.astype(np.float64), N, p, r, budget,
                             float(np.float32(alpha)))
        assert np.array_equal(to_np(kept), want), (f, budget, alpha)


def test_fused_selection_fallback_matches_steps():
    """V norms that crowd one bin of the VaN map: the fused pass's 512-thread
    selection takes the exact window search (the step kernels' 1024-thread
    block as well in one slab, direct ranking in the other); indices and
    bytes must agree bit for bit."""
    S, f, gh, gw, D = 2, 256, 4, 4, 64
    w = synth.Workload("crowded", 1, S, D, "f32", gh, gw, f, 128 * gh * gw, 0.5, seed=3)
    p, N = w.p, w.n_tokens
    K, V = synth.host_generate(w)
    rng = np.random.default_rng(9)
    r = oracle.recent_frames(f)
    n_past = N - r * p
    for s, n_cluster in ((0, 2600), (1, 800)):
        u = V[s, :n_past] / np.linalg.norm(V[s, :n_past], axis=1, keepdims=True)
        norm = rng.uniform(0.2, 0.5, n_past)
        idx = rng.permutation(n_past)
        norm[idx[:n_cluster]] = 1.0 + rng.integers(0, 4000, n_cluster) * 1e-6
        norm[idx[n_cluster:n_cluster + 300]] = rng.uniform(2.0, 100.0, 300)
        norm[idx[n_cluster + 300]] = 1000.0
        V[s, :n_past] = (u * norm[:, None]).astype(np.float32)

    def make_cache():
        c = PingPongCache(S, N, D, "f32", patch_ids=True)
        c.k[0] = to_dev(K, "f32")
        c.v[0] = to_dev(V, "f32")
        return c

    (kp, cp), (ks, cs) = _run_both(w, 1, make_cache, pid_valid=False, passes=1)
    B = w.budget
    assert torch.equal(kp, ks)
    assert torch.equal(cp.v[1, :, :B], cs.v[1, :, :B])


def test_invalid_arguments_are_rejected():
    S, f, gh, gw, D = 2, 8, 4, 4, 64
    p, N = gh * gw, f * gh * gw
    init_for(S, N, D, p, "f32")
    cache = host_case(S, f, gh, gw, D, "f32", seed=1)
    kept = torch.empty((S, N), dtype=torch.int32, device="cuda")
    k, v = cache.structs(False)
    bad = [
        dict(n_tokens=N + p),                 # above token_capacity
        dict(n_tokens=N - 1),                 # not whole frames
        dict(budget=p),                       # r p >= budget
        dict(tar_ratio=1.5),
        dict(tar_ratio=float("nan")),
        dict(head_dim=D * 2),                 # above max_head_dim
        dict(n_layers=2),                     # above max_slabs
        dict(frame_grid_w=gw * 2, n_tokens=N),  # above max_frame_tokens
    ]
    for over in bad:
        args = dict(n_layers=1, n_kv_heads=S, head_dim=D, n_tokens=N, frame_grid_h=gh,
                    frame_grid_w=gw, budget=N // 2, tar_ratio=0.5)
        args.update(over)
        with pytest.raises(ipv.IpvError) as ei:
            ipv.compress(k, v, args["n_layers"], args["n_kv_heads"], args["head_dim"],
                         args["n_tokens"], args["frame_grid_h"], args["frame_grid_w"],
                         args["budget"], args["tar_ratio"], kept)
        assert ei.value.status == ipv.IPV_EINVAL, over
        assert k.cur == 0 and v.cur == 0


def test_scratch_allocation_failure_is_reported_and_recovered():
    """ipv_init asking for more scratch than the GPU holds fails with
    IPV_ENOMEM (no kernel runs, nothing stays allocated), leaves the library
    uninitialised, and the next ipv_init and pass work as before."""
    slabs, cap = 2_000_000, 49152  # 393 GB per score array
    free, total = torch.cuda.mem_get_info()
    assert slabs * cap * 4 > total
    with pytest.raises(ipv.IpvError) as ei:
        ipv.init(device=0, dtype="bf16", max_head_dim=128, max_frame_tokens=256, max_slabs=slabs,
                 token_capacity=cap)
    assert ei.value.status == ipv.IPV_ENOMEM
    assert ipv.recent_frames(48) == -1  # not initialised
    assert torch.cuda.mem_get_info()[0] >= free - (64 << 20)  # the partial allocations were freed
    S, f, gh, gw, D = 2, 10, 4, 5, 64
    init_for(S, f * gh * gw, D, gh * gw, "bf16")
    cache = host_case(S, f, gh, gw, D, "bf16", seed=12)
    check_pass(cache, 1, S, f * gh * gw, gh, gw, 90, 0.5, pid_valid=False)


def _device_config(name, patch_ids=False):
    w = synth.CONFIGS[name]
    init_for(w.slabs_per_stream, w.n_tokens, w.head_dim, w.p, w.dtype)
    cache = PingPongCache(w.slabs_per_stream, w.n_tokens, w.head_dim, w.dtype, patch_ids=patch_ids)
    synth.device_generate(w, cache.k[0], cache.v[0])
    return w, cache


@pytest.mark.parametrize("name", ["llava", "qwen"])
def test_full_config(name):
    """Configs at full size (28 layers x 4 KV heads), every slab checked."""
    w, cache = _device_config(name, patch_ids=True)
    check_pass(cache, w.n_layers, w.n_kv_heads, w.n_tokens, w.grid_h, w.grid_w, w.budget,
               w.tar_ratio, pid_valid=False)


def test_passthrough_full_shape():
    """A budget of every cached token at the LLaVA shape (112 slabs x 9408
    tokens): nothing is evicted, so the pass leaves the cache where it is and
    the kept indices are 0..N-1, through ipv_compress and ipv_select alike."""
    w, cache = _device_config("llava", patch_ids=True)
    N, S = w.n_tokens, w.slabs_per_stream
    k_before = cache.k_live.clone()
    check_pass(cache, w.n_layers, w.n_kv_heads, N, w.grid_h, w.grid_w, N, w.tar_ratio, pid_valid=False)
    assert torch.equal(cache.k_live, k_before)
    kept = torch.full((S, N), -7, dtype=torch.int32, device="cuda")
    tar = torch.zeros((S, N), dtype=torch.float32, device="cuda")
    ipv.select(tar, tar, S, N, w.grid_h, w.grid_w, N, w.tar_ratio, kept)
    assert torch.equal(kept, torch.arange(N, dtype=torch.int32, device="cuda").expand(S, N))


def test_streaming_run():
    """1 h at 1 fps at the LLaVA shape (Algorithm 1's loop): 16 frames
    appended per step through ipv_append_frames (patch ids and frame ids
    numbered on the device), a pass whenever the cache holds 9408 tokens.
    Every pass keeps the invariants; 10 evenly spaced passes of the 223 are
    checked against the oracle on every slab (past rows then carry patch and
    frame ids from earlier passes, and the ids must follow their rows)."""
    w = synth.CONFIGS["stream"]
    S, p, D, N, nf = w.slabs_per_stream, w.p, w.head_dim, w.n_tokens, w.append_frames
    init_for(S, N, D, p, w.dtype)
    cache = PingPongCache(S, N, D, w.dtype, patch_ids=True, frame_ids=True)
    gen = synth.DeviceGenerator(w, S)
    k_new = torch.empty((S, nf * p, D), dtype=cache.k.dtype, device="cuda")
    v_new = torch.empty_like(k_new)
    kept = torch.empty((S, w.budget), dtype=torch.int32, device="cuda")
    n_passes = (w.stream_frames - w.n_frames) // nf + 1
    check_at = set(np.linspace(0, n_passes - 1, 10).round().astype(int).tolist())
    r = ipv.recent_frames(w.n_frames)
    passes = frames = 0
    while frames < w.stream_frames:
        assert w.stream_frames - frames >= nf  # 3600 frames are 225 blocks of 16
        gen.fill(k_new, v_new, 0, nf)
        k, v = cache.structs(pid_valid=True)
        ipv.append_frames(k, v, k_new, v_new, w.n_layers, w.n_kv_heads, D, cache.n_tokens, nf,
                          w.grid_h, w.grid_w)
        cache.n_tokens += nf * p
        frames += nf
        if cache.n_tokens >= N:
            assert cache.n_tokens == N
            if passes in check_at:
                check_pass(cache, w.n_layers, w.n_kv_heads, N, w.grid_h, w.grid_w,
                           w.budget, w.tar_ratio, pid_valid=True)
                newest = cache.fid[cache.cur, :, w.budget - 1]
                assert torch.all(newest == frames - 1)  # device numbering followed the stream
            else:
                cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, w.budget,
                               w.tar_ratio, kept, pid_valid=True)
                kn = kept
                assert torch.all(kn[:, 1:] > kn[:, :-1])
                assert torch.equal(kn[:, -r * p:], torch.arange(N - r * p, N, device="cuda",
                                                                dtype=torch.int32).expand(S, -1))
            passes += 1
    assert passes == n_passes == 223 and len(check_at) == 10


def test_large_config_sampled():
    """8 streams x 80 layers x 8 KV heads, 32768 -> 24576 tokens (~86 GB of
    K/V plus the second ping-pong half). 64 sampled slabs checked, 8 from
    each stream."""
    w = synth.CONFIGS["large"]
    S = w.n_slabs
    need = 2 * 2 * S * w.n_tokens * w.head_dim * 2 + 3 * S * w.n_tokens * 4 + (8 << 30)
    free, _ = torch.cuda.mem_get_info()
    if free < need:
        pytest.skip(f"needs {need / 2**30:.0f} GiB free, {free / 2**30:.0f} GiB available")
    init_for(S, w.n_tokens, w.head_dim, w.p, w.dtype)
    cache = PingPongCache(S, w.n_tokens, w.head_dim, w.dtype, patch_ids=False)
    per = w.slabs_per_stream
    for st in range(w.n_streams):
        synth.device_generate(w, cache.k[0, st * per:(st + 1) * per],
                              cache.v[0, st * per:(st + 1) * per], stream=st)
    rng = np.random.default_rng(1)
    sample = np.sort(np.concatenate([st * per + rng.choice(per, 8, replace=False)
                                     for st in range(w.n_streams)]))
    try:
        check_pass(cache, w.n_streams * w.n_layers, w.n_kv_heads, w.n_tokens, w.grid_h, w.grid_w,
                   w.budget, w.tar_ratio, pid_valid=False, slabs=sample)
    finally:
        del cache
        torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype,budget,alpha", [("bf16", 30001, 0.5), ("f32", 36864, 0.3)])
def test_max_tokens(dtype, budget, alpha):
    """n_tokens = IPV_MAX_TOKENS (192 frames of 16 x 16, r = 24): the largest
    selection the library takes, with 43008 past tokens, too many for VaN to
    sit in shared memory beside TaR, so the VaN stage reads it from L2; a
    ragged and a whole-frame budget; then the compacted cache with 16 new
    frames appended (patch ids carried) at the same size."""
    S, gh, gw, D = 2, 16, 16, 128
    p = gh * gw
    f = ipv.MAX_TOKENS // p
    N = f * p
    assert N == ipv.MAX_TOKENS
    init_for(S, N, D, p, dtype)
    assert ipv.recent_frames(f) == 24
    w = synth.Workload("max", 1, S, D, dtype, gh, gw, f, budget, alpha, seed=77)
    cache = PingPongCache(S, N, D, dtype, patch_ids=True)
    gen = synth.DeviceGenerator(w, S)  # the oracle reads the generated bytes back
    gen.fill(cache.k[0], cache.v[0], 0, f)
    check_pass(cache, 1, S, N, gh, gw, budget, alpha, pid_valid=False)
    if budget % p:
        return  # a ragged budget leaves no whole-frame cache to append to
    n_new = (N - budget) // p
    gen.fill(cache.k_live, cache.v_live, budget, n_new)
    cache.pid_live[:, budget:N] = torch.arange(p, dtype=torch.int16, device="cuda").repeat(n_new)
    check_pass(cache, 1, S, N, gh, gw, budget, alpha, pid_valid=True)


def _run_both(w, L, make_cache, pid_valid, passes=1):
    """Run `passes` passes with the fused kernel and with the step kernels on
    identical inputs; return both (kept, cache) results."""
    out = []
    for single in (True, False):
        init_for(w_slabs(w, L), w.n_tokens, w.head_dim, w.p, w.dtype, single_kernel=single)
        cache = make_cache()
        kept = torch.empty((cache.n_slabs, w.budget), dtype=torch.int32, device="cuda")
        for _ in range(passes):
            cache.cur = 0  # the same source half every time
            k, v = cache.structs(pid_valid=pid_valid)
            ipv.compress(k, v, L, w.n_kv_heads, w.head_dim, w.n_tokens, w.grid_h, w.grid_w,
                         w.budget, w.tar_ratio, kept)
        cache.cur = k.cur
        torch.cuda.synchronize()
        assert ipv.device_error() == 0
        out.append((kept.clone(), cache))
        ipv.shutdown()
    return out


def w_slabs(w, L):
    return L * w.n_kv_heads


def _fresh_cache(w):
    def make_cache():
        c = PingPongCache(w.slabs_per_stream, w.n_tokens, w.head_dim, w.dtype, patch_ids=True)
        if w.dtype == "f32":
            K, V = synth.host_generate(w)
            c.k[0] = to_dev(K, w.dtype)
            c.v[0] = to_dev(V, w.dtype)
        else:
            synth.device_generate(w, c.k[0], c.v[0])
        c.k[1].fill_(-7.0)
        c.v[1].fill_(-7.0)
        c.pid[1].fill_(-1)
        return c
    return make_cache


FUSED_SHAPES = {
    # name: (layers, KV heads, head_dim, dtype, grid, frames, budget frames, alpha)
    "ragged_items": (3, 5, 128, "bf16", (13, 11), 24, 17, 0.45),  # p = 143: items of 15 and 16 patches
    "one_patch": (2, 3, 64, "bf16", (1, 1), 40, 30, 0.5),          # p = 1: one score item per slab
    "wide_rows_f32": (2, 2, 512, "f32", (6, 7), 16, 11, 0.6),      # 2 KB rows: fewer patches per item
    "many_slabs": (40, 8, 64, "bf16", (4, 4), 32, 20, 0.3),       # 320 slabs: owners take several
    "alpha_extremes0": (2, 4, 96, "bf16", (5, 5), 20, 12, 0.0),
    "alpha_extremes1": (2, 4, 96, "bf16", (5, 5), 20, 12, 1.0),
}


@pytest.mark.parametrize("name", ["llava", "qwen", "tiny"] + sorted(FUSED_SHAPES))
def test_fused_matches_steps(name):
    """The fused kernel and the four step kernels run the same device
    arithmetic: indices, compacted rows and patch ids are bit-identical; the
    fused result also passes the oracle checks."""
    if name in FUSED_SHAPES:
        L, H, D, dt, (gh, gw), f, bf, alpha = FUSED_SHAPES[name]
        w = synth.Workload(name, L, H, D, dt, gh, gw, f, bf * gh * gw, alpha, seed=len(name))
    else:
        w = synth.CONFIGS[name]
    L = w.n_layers
    (kp, cp), (ks, cs) = _run_both(w, L, _fresh_cache(w), pid_valid=False, passes=2)
    B = w.budget
    assert torch.equal(kp, ks)
    assert cp.cur == cs.cur == 1
    assert torch.equal(cp.k[1, :, :B], cs.k[1, :, :B])
    assert torch.equal(cp.v[1, :, :B], cs.v[1, :, :B])
    assert torch.equal(cp.pid[1, :, :B], cs.pid[1, :, :B])
    if w.n_slabs * w.n_tokens <= 400_000:  # small enough for the oracle
        init_for(w_slabs(w, L), w.n_tokens, w.head_dim, w.p, w.dtype, single_kernel=True)
        try:
            cache = _fresh_cache(w)()
            check_pass(cache, L, w.n_kv_heads, w.n_tokens, w.grid_h, w.grid_w, B, w.tar_ratio,
                       pid_valid=False)
        finally:
            torch.cuda.synchronize()
            ipv.shutdown()


def test_fused_falls_back_for_a_compacted_cache():
    """A live half with patch ids (a cache compacted before) goes through the
    step kernels under single_kernel = 1: the result equals the step path's."""
    S, f, gh, gw, D = 24, 16, 7, 7, 128
    w = synth.Workload("case", 1, S, D, "bf16", gh, gw, f, 500, 0.5, seed=21)
    p, N = w.p, w.n_tokens
    K, V = synth.host_generate(w)
    r = oracle.recent_frames(f)
    n_past = N - r * p
    perm = np.random.default_rng(4).permutation(n_past)
    K[:, :n_past], V[:, :n_past] = K[:, perm], V[:, perm]
    pid = np.tile((np.arange(N) % p).astype(np.uint16), (S, 1))
    pid[:, :n_past] = (perm % p).astype(np.uint16)

    def make_cache():
        c = PingPongCache(S, N, D, "bf16", patch_ids=True)
        c.k[0] = to_dev(K, "bf16")
        c.v[0] = to_dev(V, "bf16")
        c.pid[0] = torch.from_numpy(pid.view(np.int16)).cuda()
        return c

    (kp, cp), (ks, cs) = _run_both(w, 1, make_cache, pid_valid=True, passes=3)
    B = w.budget
    assert torch.equal(kp, ks)
    assert torch.equal(cp.k[1, :, :B], cs.k[1, :, :B])
    assert torch.equal(cp.pid[1, :, :B], cs.pid[1, :, :B])
