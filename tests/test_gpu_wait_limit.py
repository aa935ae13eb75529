"""Failure detection of the fused pass without a GPU fault: every wait in
it is bounded. With a one-poll limit the waits for data that is not ready
yet (a slab's scores before its selection, a selection before the slab's
compaction) give up, set their bits in the device error word, and the pass
ends; the host reads the bits, the context stays usable, and the next pass
(default limit) starts from clean counters and gives the same result as
before the failure."""
import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2506_15745_gb300 import ipv  # noqa: E402
from paper_2506_15745_gb300.cache import PingPongCache  # noqa: E402


def test_short_wait_limit_reports_and_recovers():
    w = synth.CONFIGS["llava"].scaled(n_layers=8, n_kv_heads=4, head_dim=128, n_frames=24,
                                      budget=16 * 196, seed=4)
    S, N, C, D = w.n_slabs, w.n_tokens, w.budget, w.head_dim
    ipv.init(device=0, dtype=w.dtype, max_head_dim=D, max_frame_tokens=w.p, max_slabs=S,
             token_capacity=N, single_kernel=True)
    try:
        cache = PingPongCache(S, N, D, w.dtype, patch_ids=False)
        synth.device_generate(w, cache.k[0], cache.v[0])

        def one_pass():
            k, v = cache.structs(pid_valid=False)
            k.cur = v.cur = 0
            kept = torch.full((S, C), -1, dtype=torch.int32, device="cuda")
            ipv.compress(k, v, w.n_layers, w.n_kv_heads, D, N, w.grid_h, w.grid_w, C,
                         w.tar_ratio, kept)
            torch.cuda.synchronize()
            return kept.cpu().numpy(), cache.k[1, :, :C].clone()

        kept0, k0 = one_pass()
        assert ipv.device_error() == 0
        assert np.all(np.diff(kept0, axis=1) > 0)

        ipv.set_wait_limit(1)          # waits give up after one poll
        one_pass()                     # results invalid, but the pass ends
        err = ipv.device_error()
        assert err != 0 and (err & ~3) == 0, err
        assert ipv.device_error() == 0  # reading clears the word

        ipv.set_wait_limit(0)          # back to the default
        kept1, k1 = one_pass()
        assert ipv.device_error() == 0
        assert np.array_equal(kept0, kept1) and torch.equal(k0, k1)
    finally:
        torch.cuda.synchronize()
        ipv.shutdown()
