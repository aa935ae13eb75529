"""ipv_compress_static: the pass for callers that cannot allocate device memory.

Its working memory is a fixed array in the library's device image, so it needs
neither cudaMalloc nor ipv_init. These tests call it through the C ABI and
compare it with ipv_compress on the same inputs, on two calls in a row with
different shapes (the second call finds the first call's leftovers in the
shared array). The file name sorts last, so a run that stops at the first
failure has run every other test before this one.
"""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2506_15745_gb300 import ipv  # noqa: E402
from paper_2506_15745_gb300.cache import PingPongCache  # noqa: E402


def _llava_case():
    w = synth.CONFIGS["llava"]
    cache = PingPongCache(w.slabs_per_stream, w.n_tokens, w.head_dim, w.dtype, patch_ids=True)
    synth.device_generate(w, cache.k[0], cache.v[0])
    return w, cache, False


def _qwen_case():
    """The Qwen2-VL-7B shape: about 29.4 MB of the 32 MiB array, the pass
    closest to the limit that the header promises to accept."""
    w = synth.CONFIGS["qwen"]
    cache = PingPongCache(w.slabs_per_stream, w.n_tokens, w.head_dim, w.dtype, patch_ids=True)
    synth.device_generate(w, cache.k[0], cache.v[0])
    return w, cache, False


def _f32_case():
    """fp32 storage: 3 layers x 2 heads, D=64, 6x6 patches, 24 frames."""
    w = synth.Workload("f32case", 3, 2, 64, "f32", 6, 6, 24, 600, 0.6, seed=7)
    K, V = synth.host_generate(w)
    cache = PingPongCache(w.slabs_per_stream, w.n_tokens, w.head_dim, w.dtype, patch_ids=True)
    cache.k[0] = torch.from_numpy(K).cuda()
    cache.v[0] = torch.from_numpy(V).cuda()
    return w, cache, False


def _shuffled_case():
    """2 layers x 3 heads, D=64 bf16, 7x7 patches, 16 frames, past rows
    shuffled together with their patch ids (a cache compacted before)."""
    w = synth.Workload("shuffled", 2, 3, 64, "bf16", 7, 7, 16, 500, 0.4, seed=5)
    K, V = synth.host_generate(w)
    N, p = w.n_tokens, w.p
    n_past = N - oracle.recent_frames(w.n_frames) * p
    perm = np.random.default_rng(2).permutation(n_past)
    K[:, :n_past], V[:, :n_past] = K[:, perm], V[:, perm]
    pid = np.tile((np.arange(N) % p).astype(np.uint16), (w.slabs_per_stream, 1))
    pid[:, :n_past] = (perm % p).astype(np.uint16)
    cache = PingPongCache(w.slabs_per_stream, N, w.head_dim, w.dtype, patch_ids=True)
    cache.k[0] = torch.from_numpy(K.view(np.int16)).cuda().view(torch.bfloat16)
    cache.v[0] = torch.from_numpy(V.view(np.int16)).cuda().view(torch.bfloat16)
    cache.pid[0] = torch.from_numpy(pid.view(np.int16)).cuda()
    return w, cache, True


def _run_pair(w, cache, pid_valid):
    """ipv_compress, then ipv_compress_static on the same source half;
    returns both results (kept indices, compacted K, V and patch ids)."""
    S, N, B, D = w.slabs_per_stream, w.n_tokens, w.budget, w.head_dim
    results = []
    for static in (False, True):
        cache.k[1].fill_(-3.0)
        cache.v[1].fill_(-3.0)
        cache.pid[1].fill_(-1)
        kept = torch.full((S, B), -9, dtype=torch.int32, device="cuda")
        k, v = cache.structs(pid_valid=pid_valid)
        k.cur = v.cur = 0
        if static:
            ipv.compress_static(k, v, w.dtype, N, 0, w.n_layers, w.n_kv_heads, D, N, w.grid_h,
                                w.grid_w, B, w.tar_ratio, kept)
        else:
            ipv.init(device=0, dtype=w.dtype, max_head_dim=D, max_frame_tokens=w.p,
                     max_slabs=S, token_capacity=N)
            ipv.compress(k, v, w.n_layers, w.n_kv_heads, D, N, w.grid_h, w.grid_w, B,
                         w.tar_ratio, kept)
            torch.cuda.synchronize()
            ipv.shutdown()  # the static entry point must not depend on ipv_init
        torch.cuda.synchronize()
        assert k.cur == 1 and v.cur == 1
        results.append((kept.clone(), cache.k[1, :, :B].clone(), cache.v[1, :, :B].clone(),
                        cache.pid[1, :, :B].clone()))
    return results


def test_static_matches_compress_two_calls():
    for make in (_llava_case, _qwen_case, _shuffled_case, _f32_case):
        w, cache, pid_valid = make()
        (kc, kdc, vdc, pc), (ks, kds, vds, ps) = _run_pair(w, cache, pid_valid)
        # Indices are integer work: bit-exact. Rows are copied bytes: bit-exact.
        assert torch.equal(kc, ks), w.name
        assert torch.equal(kdc, kds) and torch.equal(vdc, vds), w.name
        assert torch.equal(pc, ps), w.name
        r = oracle.recent_frames(w.n_frames)
        kn = ks.cpu().numpy()
        assert np.all(np.diff(kn, axis=1) > 0)
        assert np.all(kn[:, -r * w.p:] == np.arange(w.n_tokens - r * w.p, w.n_tokens))
        del cache
        torch.cuda.empty_cache()


def test_static_rejects_a_pass_larger_than_its_array():
    # 448 slabs of the LLaVA shape need about 80 MB of working memory; the
    # arguments are checked before any pointer is used.
    fake = [0x100000 * (i + 1) for i in range(4)]
    k = ipv.KV.from_tensors((fake[0], fake[1]), (None, None), 0)
    v = ipv.KV.from_tensors((fake[2], fake[3]), (None, None), 0)
    with pytest.raises(ipv.IpvError) as ei:
        ipv.compress_static(k, v, "bf16", 9408, 0, 112, 4, 128, 9408, 14, 14, 6272, 0.5,
                            0x200000)
    assert ei.value.status == ipv.IPV_EINVAL
    assert "working memory" in str(ei.value)
    assert k.cur == 0 and v.cur == 0


def test_static_rejects_slab_counts_whose_byte_count_would_wrap():
    # 2^30 x 2^30 slabs of 4 tokens: the byte counts would wrap to 0 in 64
    # bits; the pass must still be rejected before anything is enqueued.
    fake = [0x100000 * (i + 1) for i in range(4)]
    k = ipv.KV.from_tensors((fake[0], fake[1]), (None, None), 0)
    v = ipv.KV.from_tensors((fake[2], fake[3]), (None, None), 0)
    with pytest.raises(ipv.IpvError) as ei:
        ipv.compress_static(k, v, "f32", 4, 0, 1 << 30, 1 << 30, 4, 4, 1, 1, 2, 0.5, 0x200000)
    assert ei.value.status == ipv.IPV_EINVAL
    assert k.cur == 0 and v.cur == 0


def test_static_passes_a_cache_within_budget_through():
    """n_tokens <= budget: kept = 0..n_tokens-1 padded with -1; the cache is
    neither copied nor flipped."""
    S, N, B, D = 6, 48, 60, 64
    cache = PingPongCache(S, 64, D, "bf16", patch_ids=True)
    cache.k[0].normal_()
    cache.v[0].normal_()
    cache.k[1].fill_(-3.0)
    before = cache.k[1].clone()
    kept = torch.full((S, B), -9, dtype=torch.int32, device="cuda")
    k, v = cache.structs(pid_valid=False)
    ipv.compress_static(k, v, "bf16", 64, 0, 3, 2, D, N, 4, 4, B, 0.5, kept)
    torch.cuda.synchronize()
    assert k.cur == 0 and v.cur == 0
    want = torch.full((S, B), -1, dtype=torch.int32)
    want[:, :N] = torch.arange(N, dtype=torch.int32)
    assert torch.equal(kept.cpu(), want)
    assert torch.equal(cache.k[1], before)


def _random_case(case):
    """A small seeded shape: element type, heads, head_dim, grid, frames,
    budget and ratio drawn at random; half the cases come compacted before
    (past rows shuffled with their patch ids)."""
    rng = np.random.default_rng(900 + case)
    dtype = ("bf16", "f32")[int(rng.integers(2))]
    L, H = int(rng.integers(1, 4)), int(rng.integers(1, 5))
    D = int(rng.choice((16, 32, 64, 128, 256)))
    gh, gw = int(rng.integers(1, 10)), int(rng.integers(1, 10))
    f = int(rng.integers(4, 25))
    r = oracle.recent_frames(f)
    budget = int(rng.integers(r * gh * gw + 1, f * gh * gw))
    alpha = float(np.float32(rng.choice([0.0, 1.0, rng.uniform(0, 1)])))
    w = synth.Workload(f"random{case}", L, H, D, dtype, gh, gw, f, budget, alpha, seed=case)
    K, V = synth.host_generate(w)
    N, p, S = w.n_tokens, w.p, w.slabs_per_stream
    cache = PingPongCache(S, N, D, dtype, patch_ids=True)
    shuffled = bool(rng.integers(2))
    if shuffled:
        n_past = N - r * p
        perm = rng.permutation(n_past)
        K[:, :n_past], V[:, :n_past] = K[:, perm], V[:, perm]
        pid = np.tile((np.arange(N) % p).astype(np.uint16), (S, 1))
        pid[:, :n_past] = (perm % p).astype(np.uint16)
        cache.pid[0] = torch.from_numpy(pid.view(np.int16)).cuda()
    if dtype == "bf16":
        cache.k[0] = torch.from_numpy(K.view(np.int16)).cuda().view(torch.bfloat16)
        cache.v[0] = torch.from_numpy(V.view(np.int16)).cuda().view(torch.bfloat16)
    else:
        cache.k[0] = torch.from_numpy(K).cuda()
        cache.v[0] = torch.from_numpy(V).cuda()
    return w, cache, shuffled


def test_static_matches_compress_on_random_shapes():
    """40 seeded shapes in a row: each call of the static entry point finds
    the previous, differently shaped call's leftovers in the shared array."""
    for case in range(40):
        w, cache, pid_valid = _random_case(case)
        (kc, kdc, vdc, pc), (ks, kds, vds, ps) = _run_pair(w, cache, pid_valid)
        assert torch.equal(kc, ks), case
        assert torch.equal(kdc, kds) and torch.equal(vdc, vds), case
        assert torch.equal(pc, ps), case
