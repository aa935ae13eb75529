"""Streaming (Algorithm 1's loop) with the steady-state step captured in CUDA
graphs: "append 6 new frames, then compress" is captured once per ping-pong
parity and replayed; frame ids are numbered on the device, so the replayed
stream must equal the eagerly launched one bit for bit (kept indices,
compacted K/V, patch and frame ids), for the raw and the pooled pass."""
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


F0, A, STEPS = 16, 6, 9           # first fill, frames appended per step, steady steps


def _setup(pooled, dtype):
    base = synth.CONFIGS["llava_pool" if pooled else "llava"]
    w = base.scaled(n_layers=2, n_kv_heads=2, head_dim=64, grid_h=7, grid_w=7, n_frames=F0,
                    budget=10 * 49, dtype=dtype, seed=21)
    K, V = synth.host_generate(w, n_frames=F0 + A * STEPS)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    def dev(a):
        t = torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if dtype == "bf16" else a)).cuda()
        return t.view(tdt)
    return w, dev(K), dev(V)


def _init(w, pooled):
    ipv.init(device=0, dtype=w.dtype, max_head_dim=w.head_dim, max_frame_tokens=w.p,
             max_slabs=w.n_slabs, token_capacity=w.n_tokens, van_pool=pooled, cv_tau=(0.3, 0.5, 0.8))


def _frames(K, p, f0, nf):
    return K[:, f0 * p:(f0 + nf) * p].contiguous()


def _structs(cache, cur):
    k = ipv.KV.from_tensors((cache.k[0], cache.k[1]), (cache.pid[0], cache.pid[1]), cur,
                            (cache.fid[0], cache.fid[1]))
    v = ipv.KV.from_tensors((cache.v[0], cache.v[1]), (None, None), cur)
    return k, v


def _first_fill(w, cache, K, V, kept):
    k, v = _structs(cache, 0)
    ipv.append_frames(k, v, _frames(K, w.p, 0, F0), _frames(V, w.p, 0, F0), w.n_layers,
                      w.n_kv_heads, w.head_dim, 0, F0, w.grid_h, w.grid_w, first_frame=100)
    ipv.compress(k, v, w.n_layers, w.n_kv_heads, w.head_dim, w.n_tokens, w.grid_h, w.grid_w,
                 w.budget, w.tar_ratio, kept)
    return k.cur


def _step(w, cache, cur, k_new, v_new, kept):
    k, v = _structs(cache, cur)
    ipv.append_frames(k, v, k_new, v_new, w.n_layers, w.n_kv_heads, w.head_dim, w.budget, A,
                      w.grid_h, w.grid_w)
    ipv.compress(k, v, w.n_layers, w.n_kv_heads, w.head_dim, w.n_tokens, w.grid_h, w.grid_w,
                 w.budget, w.tar_ratio, kept)
    return k.cur


def _snapshot(cache, cur, B, kept):
    return (kept.clone(), cache.k[cur, :, :B].clone(), cache.v[cur, :, :B].clone(),
            cache.pid[cur, :, :B].clone(), cache.fid[cur, :, :B].clone())


@pytest.mark.parametrize("pooled,dtype", [(False, "bf16"), (True, "bf16"), (False, "f32")])
def test_graph_replayed_stream_equals_eager(pooled, dtype):
    w, K, V = _setup(pooled, dtype)
    _init(w, pooled)
    B, p = w.budget, w.p
    results = []
    for use_graph in (False, True):
        cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype, patch_ids=True, frame_ids=True)
        cache.k.zero_()
        cache.v.zero_()
        kept = torch.full((w.n_slabs, B), -1, dtype=torch.int32, device="cuda")
        k_new = torch.empty_like(_frames(K, p, 0, A))
        v_new = torch.empty_like(k_new)
        cur = _first_fill(w, cache, K, V, kept)
        graphs = {}
        if use_graph:
            torch.cuda.synchronize()
            for c in (0, 1):  # one graph per ping-pong parity; capture runs nothing
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    _step(w, cache, c, k_new, v_new, kept)
                graphs[c] = g
        for t in range(STEPS):
            f0 = F0 + A * t
            k_new.copy_(_frames(K, p, f0, A))
            v_new.copy_(_frames(V, p, f0, A))
            if use_graph:
                graphs[cur].replay()
                cur = 1 - cur
            else:
                cur = _step(w, cache, cur, k_new, v_new, kept)
        torch.cuda.synchronize()
        results.append(_snapshot(cache, cur, B, kept))
    for a, b in zip(*results):
        assert torch.equal(a, b)
    kept_np = results[0][0].cpu().numpy()
    assert np.all(np.diff(kept_np, axis=1) > 0)
    fid = results[0][4].cpu().numpy()
    assert fid.max() == 100 + F0 + A * STEPS - 1          # device-side frame numbering
    assert np.all(np.diff(fid.astype(np.int64), axis=1) >= 0)


def test_append_frames_writes_rows_and_ids():
    w, K, V = _setup(False, "bf16")
    _init(w, False)
    p = w.p
    cache = PingPongCache(w.n_slabs, w.n_tokens, w.head_dim, w.dtype, patch_ids=True, frame_ids=True)
    cache.fid.fill_(-1)
    cache.fid[0, :, 99] = 41                                      # the last cached row's frame
    k, v = _structs(cache, 0)
    ipv.append_frames(k, v, _frames(K, p, 3, 2), _frames(V, p, 3, 2), w.n_layers, w.n_kv_heads,
                      w.head_dim, 100, 2, w.grid_h, w.grid_w)
    torch.cuda.synchronize()
    assert torch.equal(cache.k[0, :, 100:100 + 2 * p], _frames(K, p, 3, 2))
    assert torch.equal(cache.v[0, :, 100:100 + 2 * p], _frames(V, p, 3, 2))
    pid = cache.pid[0, :, 100:100 + 2 * p].cpu().numpy()
    fid = cache.fid[0, :, 100:100 + 2 * p].cpu().numpy()
    assert np.all(pid == np.tile(np.arange(p), 2)) and np.all(fid == np.repeat([42, 43], p))
    with pytest.raises(ipv.IpvError):                              # beyond token_capacity
        ipv.append_frames(k, v, _frames(K, p, 3, 2), _frames(V, p, 3, 2), w.n_layers, w.n_kv_heads,
                          w.head_dim, w.n_tokens - p, 2, w.grid_h, w.grid_w)
