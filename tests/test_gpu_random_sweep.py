"""GPU parity over a seeded random sweep of pass configurations.

Each case draws a shape (layers, KV heads, head_dim, element type, frame
grid, frame count), a budget of whole frames, a TaR ratio and one of the
pass's modes: per-head index sets on the step kernels (sometimes with the
recent-frame count overridden) or on the fused persistent kernel,
layer-adaptive pooled VaN (Sec. 3.2, Algorithm 2), one index set per layer
(Sec. 3.1, K[:, I, :]), both of the last two, or a variant of the ablation
table (Sec. 4), Uniform Select included. The pass runs on a fresh cache;
then, twice, whole frames (the AR continuation of the same streams) are
appended behind the survivors, by torch writes or by ipv_append_frames, and
it runs again on the compacted cache, patch and frame ids carried
(Algorithm 1's loop). Every pass is
checked against the oracle with the rules of parity.py: scores, pooled
scores and pool sizes, indices, compacted bytes and ids.
"""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2506_15745_gb300 import ipv  # noqa: E402
from paper_2506_15745_gb300.cache import PingPongCache  # noqa: E402
from test_gpu_parity import check_pass, to_dev  # noqa: E402
from test_gpu_pool import check_pooled_pass, spread_tau  # noqa: E402
from test_gpu_ablation import check_ablation_pass  # noqa: E402
from test_gpu_ablation import check_uniform_pass  # noqa: E402
from test_gpu_shared import check_shared_pass  # noqa: E402

MODES = ("heads", "heads_single_kernel", "pooled", "shared", "shared_pooled", "tar_reverse",
         "van_reverse", "tar_frame", "uniform")
ABLATIONS = ("tar_reverse", "van_reverse", "tar_frame", "uniform")
N_CASES = 1005
N_PASSES = 3


@pytest.fixture(autouse=True)
def _shutdown_after():
    yield
    torch.cuda.synchronize()
    ipv.shutdown()


def draw(case):
    """(mode, workload, r override or 0, append through ipv_append_frames) of
    one case. Budgets are whole frames, so the compacted cache takes whole
    frames again and stays a multiple of p."""
    rng = np.random.default_rng(1000 + case)
    mode = MODES[case % len(MODES)]
    dtype = ("bf16", "f32")[int(rng.integers(2))]
    es = 2 if dtype == "bf16" else 4
    L, H = int(rng.integers(1, 4)), int(rng.integers(1, 5))
    dims = (16, 32, 64, 96, 128, 160, 256, 512)
    if mode.startswith("shared"):
        dims = tuple(d for d in dims if H * d * es <= 2048)
    D = int(rng.choice(dims))
    gh, gw = int(rng.integers(1, 13)), int(rng.integers(1, 13))
    f = int(rng.integers(3, 21))
    r = oracle.recent_frames(f)
    budget_frames = int(rng.integers(r + 1, f))
    alpha = float(rng.choice([0.0, 1.0, round(float(rng.uniform(0.05, 0.95)), 3)], p=[0.15, 0.15, 0.7]))
    base = synth.CONFIGS["llava_pool" if mode.endswith("pooled") else "llava"]
    w = base.scaled(n_layers=L, n_kv_heads=H, head_dim=D, dtype=dtype, grid_h=gh, grid_w=gw,
                    n_frames=f, budget=budget_frames * gh * gw, tar_ratio=alpha, seed=case,
                    head_shared=mode.startswith("shared"))
    # an r other than the default, below the budget's frame count
    r_override = int(rng.integers(1, budget_frames)) if mode == "heads" and rng.random() < 0.4 else 0
    use_append_entry = bool(rng.integers(2))
    return mode, w, r_override, use_append_entry


def _cache(w, frame_ids):
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype, patch_ids=True,
                          frame_ids=frame_ids)
    cache.k.zero_()
    cache.v.zero_()
    return cache


def _append(cache, K, V, w, step, use_append_entry):
    """The next N - B rows of the generated streams (frames f + (step - 1) n_new
    onwards) behind the budget survivors, by torch writes or by the library's
    append entry point (which numbers frame ids on from the last cached row)."""
    p, N, B, f = w.p, w.n_tokens, w.budget, w.n_frames
    n_new = (N - B) // p
    src = slice(N + (step - 1) * n_new * p, N + step * n_new * p)
    k_new, v_new = to_dev(K[:, src], w.dtype), to_dev(V[:, src], w.dtype)
    if use_append_entry:
        k, v = cache.structs(pid_valid=True)
        ipv.append_frames(k, v, k_new, v_new, w.n_layers, w.n_kv_heads, w.head_dim, B, n_new,
                          w.grid_h, w.grid_w)
        return
    c = cache.cur
    f0 = f + (step - 1) * n_new
    cache.k[c, :, B:N] = k_new
    cache.v[c, :, B:N] = v_new
    cache.pid[c, :, B:N] = torch.arange(p, dtype=torch.int16, device="cuda").repeat(n_new)
    if cache.fid is not None:
        cache.fid[c, :, B:N] = torch.arange(f0, f0 + n_new, dtype=torch.int32,
                                            device="cuda").repeat_interleave(p)


@pytest.mark.parametrize("case", range(N_CASES))
def test_random_pass_fresh_then_compacted(case):
    mode, w, r_override, use_append_entry = draw(case)
    p, N, B, L, H, D = w.p, w.n_tokens, w.budget, w.n_layers, w.n_kv_heads, w.head_dim
    K, V = synth.host_generate(w, n_frames=w.n_frames + (N_PASSES - 1) * (N - B) // p)
    pooled = mode.endswith("pooled")
    tau = (0.0, 0.0, 0.0)
    if pooled:
        van_all = (oracle.van_all_shared(V[:, :N], H, N) if w.head_shared
                   else oracle.van_all(V[:, :N], N))
        cvs = oracle.van_pool(van_all, 1 if w.head_shared else H, w.grid_h, w.grid_w, (0, 0, 0))[2]
        tau = spread_tau(cvs, w.cv_tau)
    ablation = mode if mode in ABLATIONS else "none"
    ipv.init(device=0, dtype=w.dtype, recent_frames=r_override, max_head_dim=D,
             max_frame_tokens=p, max_slabs=w.n_slabs, token_capacity=N,
             single_kernel=mode == "heads_single_kernel", van_pool=pooled, cv_tau=tau,
             head_shared=w.head_shared, ablation=ablation)
    if r_override:
        assert ipv.recent_frames(w.n_frames) == r_override
    cache = _cache(w, frame_ids=pooled or w.head_shared or ablation != "none")
    cache.k[0, :, :N] = to_dev(K[:, :N], w.dtype)
    cache.v[0, :, :N] = to_dev(V[:, :N], w.dtype)
    for step in range(N_PASSES):
        pid_valid = step > 0
        if pid_valid:
            _append(cache, K, V, w, step, use_append_entry)
        if w.head_shared:
            check_shared_pass(cache, w, N, pid_valid, tau=tau if pooled else None)
        elif pooled:
            check_pooled_pass(cache, w, N, tau, pid_valid)
        elif ablation == "uniform":
            check_uniform_pass(cache, w, N, pid_valid, w.n_slabs)
        elif ablation != "none":
            check_ablation_pass(cache, w, N, ablation, pid_valid)
        else:
            check_pass(cache, L, H, N, w.grid_h, w.grid_w, B, w.tar_ratio, pid_valid)
