"""Slabs are independent: passes over layer-aligned slab ranges of a cache
(what a caller does to overlap host copies with compute) give exactly the
whole pass's indices and compacted rows, for per-head and per-layer index
sets."""
import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2506_15745_gb300 import ipv  # noqa: E402
from paper_2506_15745_gb300.cache import PingPongCache  # noqa: E402


@pytest.fixture(autouse=True)
def _shutdown_after():
    yield
    torch.cuda.synchronize()
    ipv.shutdown()


@pytest.mark.parametrize("shared", [False, True])
def test_layer_chunks_equal_the_whole_pass(shared):
    w = synth.CONFIGS["llava"].scaled(n_layers=7, n_kv_heads=4, head_dim=64, grid_h=7, grid_w=7,
                                      n_frames=16, budget=10 * 49, seed=8)
    S, N, C, D, H = w.n_slabs, w.n_tokens, w.budget, w.head_dim, w.n_kv_heads
    ipv.init(device=0, dtype=w.dtype, max_head_dim=D, max_frame_tokens=w.p, max_slabs=S,
             token_capacity=N, head_shared=shared)
    cache = PingPongCache(S, N, D, w.dtype, patch_ids=False)
    synth.device_generate(w, cache.k[0], cache.v[0])
    rows = w.n_layers if shared else S
    outs = []
    for bounds in ([(0, 7)], [(0, 2), (2, 3), (3, 7)]):   # layer ranges
        cache.k[1].zero_()
        cache.v[1].zero_()
        kept = torch.full((rows, C), -1, dtype=torch.int32, device="cuda")
        for l0, l1 in bounds:
            lo, hi = l0 * H, l1 * H
            k = ipv.KV.from_tensors((cache.k[0, lo:hi], cache.k[1, lo:hi]), (None, None), 0)
            v = ipv.KV.from_tensors((cache.v[0, lo:hi], cache.v[1, lo:hi]), (None, None), 0)
            r0, r1 = (l0, l1) if shared else (lo, hi)
            ipv.compress(k, v, l1 - l0, H, D, N, w.grid_h, w.grid_w, C, w.tar_ratio, kept[r0:r1])
        torch.cuda.synchronize()
        outs.append((kept.clone(), cache.k[1, :, :C].clone(), cache.v[1, :, :C].clone()))
    for a, b in zip(*outs):
        assert torch.equal(a, b)
    assert (outs[0][0] >= 0).all()


def test_pass_on_a_side_stream():
    """The pass enqueued on a non-default stream (inputs written on that
    stream, the result read after synchronising it) equals the pass on the
    default stream bit for bit: every kernel of the call follows the given
    stream."""
    w = synth.CONFIGS["llava"].scaled(n_layers=3, n_kv_heads=4, head_dim=128, grid_h=7, grid_w=7,
                                      n_frames=16, budget=10 * 49, seed=9)
    S, N, C, D = w.n_slabs, w.n_tokens, w.budget, w.head_dim
    ipv.init(device=0, dtype=w.dtype, max_head_dim=D, max_frame_tokens=w.p, max_slabs=S,
             token_capacity=N)
    outs = []
    for use_side in (False, True):
        st = torch.cuda.Stream() if use_side else torch.cuda.current_stream()
        with torch.cuda.stream(st):
            cache = PingPongCache(S, N, D, w.dtype, patch_ids=True)
            synth.device_generate(w, cache.k[0], cache.v[0])
            cache.n_tokens = N
            kept = torch.full((S, C), -1, dtype=torch.int32, device="cuda")
            cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, C, w.tar_ratio, kept,
                           pid_valid=False, stream=st)
        st.synchronize()
        outs.append((kept.clone(), cache.k_live[:, :C].clone(), cache.v_live[:, :C].clone(),
                     cache.pid_live[:, :C].clone()))
    for a, b in zip(*outs):
        assert torch.equal(a, b)
    assert (outs[0][0] >= 0).all()
