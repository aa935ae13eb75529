"""The C-ABI library loads, exports every entry point include/ipv.h declares,
and rejects bad arguments on the host before touching a GPU."""
import ctypes
import os
import re

import pytest

from paper_2506_15745_gb300 import build as ipv_build
from paper_2506_15745_gb300 import ipv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ipv.h")


@pytest.fixture(scope="module")
def lib():
    ipv_build.build()
    return ipv.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ipv_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert {"ipv_init", "ipv_compress", "ipv_score", "ipv_select", "ipv_shutdown",
            "ipv_last_error"} <= set(names)
    for name in names:
        assert hasattr(lib, name), name


def test_no_torch_types_in_the_header():
    text = open(HEADER).read()
    assert "torch" not in text.lower().replace("pytorch", "") and "at::" not in text


def _kv(ptrs=(16, 32), cur=0):
    return ipv.KV.from_tensors(ptrs, (None, None), cur)


def test_status_strings(lib):
    assert lib.ipv_status_string(ipv.IPV_EINVAL) == b"IPV_EINVAL"
    assert lib.ipv_status_string(ipv.IPV_ETIMEOUT) == b"IPV_ETIMEOUT"


def test_host_checks_before_init(lib):
    k, v = _kv((0x1000, 0x2000)), _kv((0x3000, 0x4000))
    kept = 0x5000
    call = lambda **kw: lib.ipv_compress(  # noqa: E731
        ctypes.byref(kw.get("k", k)), ctypes.byref(kw.get("v", v)), kw.get("L", 28), kw.get("H", 4),
        kw.get("D", 128), kw.get("N", 9408), kw.get("gh", 14), kw.get("gw", 14),
        kw.get("budget", 6272), kw.get("alpha", 0.5), kw.get("kept", kept), None)
    assert call(N=9407) == ipv.IPV_EINVAL              # not whole frames
    assert call(L=0) == ipv.IPV_EINVAL
    assert call(alpha=1.5) == ipv.IPV_EINVAL
    assert call(alpha=float("nan")) == ipv.IPV_EINVAL
    assert call(kept=None) == ipv.IPV_EINVAL
    assert call(kept=0x5002) == ipv.IPV_EINVAL         # misaligned output
    assert call(k=_kv((0x1008, 0x2000))) == ipv.IPV_EINVAL  # misaligned cache half
    assert call(k=_kv((0x1000, 0x1000))) == ipv.IPV_EINVAL  # aliasing halves
    assert call(k=_kv((0x1000, 0x2000), cur=2)) == ipv.IPV_EINVAL
    assert b"cur" in lib.ipv_last_error()
    assert call(gh=300, gw=300) == ipv.IPV_EINVAL      # p > 65535
    assert call() == ipv.IPV_ENOINIT                   # valid, but no ipv_init yet
    assert lib.ipv_select(None, None, 1, 10, 1, 1, 5, 0.5, kept, None) == ipv.IPV_EINVAL
    assert lib.ipv_select(0x100, 0x200, 1, 10, 1, 1, 5, 0.5, kept, None) == ipv.IPV_ENOINIT
    assert lib.ipv_recent_frames(48) == -1
    ms = (ctypes.c_double * 4)()
    n = (ctypes.c_int64 * 4)()
    assert lib.ipv_profile_collect(ms, n, 10) == ipv.IPV_ENOINIT


def test_init_option_checks(lib):
    assert lib.ipv_init(None) == ipv.IPV_EINVAL
    good = dict(device=0, dtype=0, recent_frames=0, max_head_dim=128, max_frame_tokens=196,
                max_slabs=112, token_capacity=9408)
    for key, bad in [("dtype", 7), ("max_head_dim", 1024), ("max_frame_tokens", 0),
                     ("max_slabs", 0), ("token_capacity", -1), ("recent_frames", -1), ("device", -1),
                     ("van_pool", 2), ("head_shared", 2), ("ablation", 5), ("ablation", -1)]:
        opt = ipv.Options(**dict(good, **{key: bad}))
        assert lib.ipv_init(ctypes.byref(opt)) == ipv.IPV_EINVAL, key
    tau = lambda *t: (ctypes.c_float * 3)(*t)  # noqa: E731
    pooled = dict(good, van_pool=1, cv_tau=tau(0.4, 0.6, 0.9))
    for key, bad in [("single_kernel", 1), ("max_frame_tokens", ipv.MAX_POOL_FRAME_TOKENS + 1),
                     ("cv_tau", tau(0.6, 0.4, 0.9)), ("cv_tau", tau(0.4, float("nan"), 0.9))]:
        opt = ipv.Options(**dict(pooled, **{key: bad}))
        assert lib.ipv_init(ctypes.byref(opt)) == ipv.IPV_EINVAL, key


def test_van_pool_host_checks(lib):
    tau = (ctypes.c_float * 3)(0.4, 0.6, 0.9)
    call = lambda **kw: lib.ipv_van_pool(  # noqa: E731
        kw.get("van", 0x1000), kw.get("pid", None), kw.get("fid", None), kw.get("stride", 0),
        kw.get("L", 28), kw.get("H", 4), kw.get("N", 9408), kw.get("gh", 14), kw.get("gw", 14),
        kw.get("tau", tau), kw.get("out", 0x2000), kw.get("ks", None), None)
    assert call(van=None) == ipv.IPV_EINVAL
    assert call(out=0x2002) == ipv.IPV_EINVAL                   # misaligned
    assert call(N=0) == ipv.IPV_EINVAL
    assert call(N=ipv.MAX_TOKENS + 1) == ipv.IPV_EINVAL
    assert call(gh=65, gw=64) == ipv.IPV_EINVAL                 # frame above the pooling limit
    assert call(gh=1, gw=4096) == ipv.IPV_EINVAL                # bordered map too large
    assert call(pid=0x3000) == ipv.IPV_EINVAL                   # patch ids without frame ids
    assert call(pid=0x3000, fid=0x4000, stride=9407) == ipv.IPV_EINVAL
    assert call(tau=(ctypes.c_float * 3)(0.9, 0.6, 0.4)) == ipv.IPV_EINVAL
    assert call(pid=0x3000, fid=0x4000, stride=9408) == ipv.IPV_ENOINIT
    assert call() == ipv.IPV_ENOINIT


def test_frame_id_checks(lib):
    k = ipv.KV.from_tensors((0x1000, 0x2000), (None, None), 0, (0x5000, 0x5000))
    v = _kv((0x3000, 0x4000))
    assert lib.ipv_compress(ctypes.byref(k), ctypes.byref(v), 28, 4, 128, 9408, 14, 14, 6272, 0.5,
                            0x6000, None) == ipv.IPV_EINVAL    # aliasing frame-id halves
    k = ipv.KV.from_tensors((0x1000, 0x2000), (None, None), 0, (0x5000, 0x5002))
    assert lib.ipv_compress(ctypes.byref(k), ctypes.byref(v), 28, 4, 128, 9408, 14, 14, 6272, 0.5,
                            0x6000, None) == ipv.IPV_EINVAL    # misaligned frame ids


def test_init_without_gpu_fails_cleanly(lib):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    opt = ipv.Options(0, 0, 0, 128, 196, 112, 9408)
    assert lib.ipv_init(ctypes.byref(opt)) == ipv.IPV_ECUDA
    assert lib.ipv_last_error().startswith(b"IPV_ECUDA")
