"""GPU parity of step (iii) alone over seeded random score distributions.

ipv_select and the oracle's selection (Sec. 3.3; Algorithm 1 steps 3-5) get
the same fp32 TaR and VaN rows and must return the same kept indices, bit for
bit. Shapes span every selection kernel (past tokens up to 9216, up to 16384
and above, to 40000); the scores mix uniform and wide-range values, heavy and
frame-like ties, tight clusters, values over many decades, NaN, infinities,
signed zeros and all-NaN rows.
"""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2506_15745_gb300 import ipv  # noqa: E402

N_CASES = 400


def _scores(rng, S, N):
    rows = []
    for _ in range(2):  # TaR, VaN
        kind = int(rng.integers(0, 8))
        if kind == 0:
            x = rng.uniform(-1, 1, (S, N))
        elif kind == 1:
            x = rng.normal(0, 1, (S, N)) * 10.0 ** rng.uniform(-20, 20)
        elif kind == 2:
            x = rng.integers(-3, 4, (S, N)) / 3.0
        elif kind == 3:
            x = 1.0 + rng.integers(0, 50, (S, N)) * 1e-7
        elif kind == 4:
            x = 10.0 ** rng.uniform(-40, 38, (S, N))
        elif kind == 5:
            x = rng.uniform(0, 3, (S, N))
            x[:, ::int(rng.integers(2, 9))] = x[0, 0]
        elif kind == 6:
            x = np.repeat(rng.normal(0, 1, (S, N // 16 + 1)), 16, axis=1)[:, :N]
        else:
            x = rng.uniform(-5, 5, (S, N)) * (rng.random((S, N)) < 0.5)
        x = x.astype(np.float32)
        m = rng.random((S, N))
        x[m < rng.uniform(0, 0.05)] = np.nan
        x[(m > 0.99) & (rng.random((S, N)) < 0.3)] = np.inf
        x[(m > 0.995) & (rng.random((S, N)) < 0.3)] = -np.inf
        if rng.random() < 0.2:
            x[m < 0.02] = -0.0
        if rng.random() < 0.1:
            x[:] = np.nan
        rows.append(x)
    return rows


def _case(case):
    rng = np.random.default_rng(70000 + case)
    p = int(rng.choice([1, 2, 4, 16, 64, 196]))
    n_past = int(rng.choice([rng.integers(1, 2000), rng.integers(2000, 9300), rng.integers(9200, 16500),
                             rng.integers(16300, 28800), rng.integers(28600, 40000)]))
    f = max(3, (n_past // p) * 8 // 7 + 1)
    if f * p > ipv.MAX_TOKENS:
        f = ipv.MAX_TOKENS // p
    N = f * p
    r = oracle.recent_frames(f)
    S = int(rng.integers(1, 5))
    budget = int(rng.integers(r * p + 1, N + 1))
    alpha = float(np.float32(rng.choice([0.0, 1.0, rng.uniform(0, 1)])))
    tar, van = _scores(rng, S, N)
    return S, N, p, r, budget, alpha, tar, van


@pytest.mark.parametrize("block", range(8))
def test_select_matches_oracle_on_random_scores(block):
    per = N_CASES // 8
    for case in range(block * per, (block + 1) * per):
        S, N, p, r, budget, alpha, tar, van = _case(case)
        ipv.init(device=0, dtype="f32", max_head_dim=64, max_frame_tokens=p, max_slabs=S,
                 token_capacity=N)
        try:
            kept = torch.empty((S, budget), dtype=torch.int32, device="cuda")
            ipv.select(torch.from_numpy(tar).cuda(), torch.from_numpy(van).cuda(), S, N, 1, p, budget,
                       alpha, kept)
            got = kept.cpu().numpy()
        finally:
            torch.cuda.synchronize()
            ipv.shutdown()
        if budget >= N:
            want = np.array([list(range(N)) + [-1] * (budget - N)] * S, np.int32)
        else:
            want = oracle.select(tar.astype(np.float64), van.astype(np.float64), N, p, r, budget, alpha)
        assert np.array_equal(got, want), (case, S, N, p, budget, alpha)


def test_select_on_more_slabs_than_sms():
    """Slabs above the register kernels' size, more of them than the GPU has
    SMs: the keys-in-shared-memory kernel then runs one block per SM, each
    taking slabs in turn. Every slab must match the oracle."""
    rng = np.random.default_rng(91)
    S, p = 300, 4
    N = 20000
    r = oracle.recent_frames(N // p)
    budget = 15001
    alpha = float(np.float32(0.4))
    tar, van = _scores(rng, S, N)
    ipv.init(device=0, dtype="f32", max_head_dim=64, max_frame_tokens=p, max_slabs=S, token_capacity=N)
    try:
        kept = torch.empty((S, budget), dtype=torch.int32, device="cuda")
        ipv.select(torch.from_numpy(tar).cuda(), torch.from_numpy(van).cuda(), S, N, 1, p, budget, alpha, kept)
        got = kept.cpu().numpy()
    finally:
        torch.cuda.synchronize()
        ipv.shutdown()
    want = oracle.select(tar.astype(np.float64), van.astype(np.float64), N, p, r, budget, alpha)
    assert np.array_equal(got, want)
