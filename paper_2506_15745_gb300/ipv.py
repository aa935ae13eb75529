"""Python binding of libipv.so (include/ipv.h): argument marshalling only.

Every step of the compression pass runs in the library's CUDA kernels; this
module converts torch tensors to device pointers and status codes to
exceptions. PyTorch supplies device memory and streams. There is no CPU
fallback: if libipv.so is missing, every call raises.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libipv.so")

IPV_OK, IPV_EINVAL, IPV_ENOINIT, IPV_ENOMEM, IPV_ECUDA, IPV_ETIMEOUT = range(6)
IPV_BF16, IPV_F32 = 0, 1
ABLATIONS = {"none": 0, "tar_reverse": 1, "van_reverse": 2, "tar_frame": 3, "uniform": 4}
NUM_KERNELS = 7
KERNEL_NAMES = ("recent_mean", "score", "select", "gather", "fused", "pool", "combine")
MAX_TOKENS = 49152
MAX_POOL_FRAME_TOKENS = 4096


class IpvError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(message)
        self.status = status


class Options(ctypes.Structure):
    _fields_ = [("device", ctypes.c_int), ("dtype", ctypes.c_int),
                ("recent_frames", ctypes.c_int), ("max_head_dim", ctypes.c_int),
                ("max_frame_tokens", ctypes.c_int), ("max_slabs", ctypes.c_int64),
                ("token_capacity", ctypes.c_int64), ("single_kernel", ctypes.c_int),
                ("van_pool", ctypes.c_int), ("cv_tau", ctypes.c_float * 3),
                ("head_shared", ctypes.c_int), ("ablation", ctypes.c_int)]


class KV(ctypes.Structure):
    """ipv_kv: the two halves of one ping-pong cache tensor (K or V)."""
    _fields_ = [("buf", ctypes.c_void_p * 2), ("patch_id", ctypes.c_void_p * 2),
                ("cur", ctypes.c_int), ("frame_id", ctypes.c_void_p * 2)]

    @classmethod
    def from_tensors(cls, halves, patch_ids=(None, None), cur: int = 0,
                     frame_ids=(None, None)) -> "KV":
        kv = cls()
        for h in range(2):
            kv.buf[h] = _ptr(halves[h])
            kv.patch_id[h] = _ptr(patch_ids[h])
            kv.frame_id[h] = _ptr(frame_ids[h])
        kv.cur = cur
        return kv


_lib = None


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def load():
    """The loaded libipv.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(LIB_PATH)
        P, I64, I32, F = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float
        KVP = ctypes.POINTER(KV)
        lib.ipv_init.argtypes = [ctypes.POINTER(Options)]
        lib.ipv_shutdown.argtypes = []
        lib.ipv_shutdown.restype = None
        lib.ipv_compress.argtypes = [KVP, KVP, I32, I32, I32, I64, I32, I32, I64, F, P, P]
        lib.ipv_score.argtypes = [KVP, KVP, I32, I32, I32, I64, I32, I32, P, P, P]
        lib.ipv_select.argtypes = [P, P, I64, I64, I32, I32, I64, F, P, P]
        lib.ipv_recent_frames.argtypes = [I64]
        lib.ipv_recent_frames.restype = I32
        lib.ipv_last_error.argtypes = []
        lib.ipv_last_error.restype = ctypes.c_char_p
        lib.ipv_status_string.argtypes = [I32]
        lib.ipv_status_string.restype = ctypes.c_char_p
        lib.ipv_profile_enable.argtypes = [I32]
        lib.ipv_profile_collect.argtypes = [ctypes.POINTER(ctypes.c_double),
                                            ctypes.POINTER(ctypes.c_int64), I32]
        lib.ipv_device_error.argtypes = [ctypes.POINTER(ctypes.c_uint32)]
        lib.ipv_compress_static.argtypes = [KVP, KVP, I32, I64, I32, I32, I32, I32, I64, I32, I32,
                                            I64, F, P, P]
        lib.ipv_van_pool.argtypes = [P, P, P, I64, I32, I32, I64, I32, I32,
                                     ctypes.POINTER(ctypes.c_float), P, P, P]
        lib.ipv_set_wait_limit.argtypes = [I64]
        lib.ipv_append_frames.argtypes = [KVP, KVP, P, P, I32, I32, I32, I64, I32, I32, I32,
                                          ctypes.c_uint32, P]
        for name in ("ipv_init", "ipv_compress", "ipv_score", "ipv_select",
                     "ipv_profile_enable", "ipv_profile_collect", "ipv_device_error",
                     "ipv_compress_static", "ipv_van_pool", "ipv_append_frames",
                     "ipv_set_wait_limit"):
            getattr(lib, name).restype = I32
        _lib = lib
    return _lib


def _check(status: int):
    if status != IPV_OK:
        raise IpvError(status, load().ipv_last_error().decode())


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def last_error() -> str:
    return load().ipv_last_error().decode()


def init(*, device: int = 0, dtype: str = "bf16", recent_frames: int = 0, max_head_dim: int,
         max_frame_tokens: int, max_slabs: int, token_capacity: int,
         single_kernel: bool = False, van_pool: bool = False,
         cv_tau=(0.0, 0.0, 0.0), head_shared: bool = False, ablation: str = "none") -> None:
    """ipv_init. van_pool: the VaN stage ranks layer-adaptive pooled VaN with
    pool size g(CV) from the thresholds cv_tau (Sec. 3.2, Algorithm 2).
    head_shared: one index set per layer for all its KV heads (Sec. 3.1).
    ablation: "tar_reverse", "van_reverse", "tar_frame" or "uniform" (Sec. 4 ablations)."""
    opt = Options(device, IPV_BF16 if dtype == "bf16" else IPV_F32, recent_frames, max_head_dim,
                  max_frame_tokens, max_slabs, token_capacity, int(bool(single_kernel)),
                  int(bool(van_pool)), (ctypes.c_float * 3)(*[float(t) for t in cv_tau]),
                  int(bool(head_shared)), ABLATIONS[ablation])
    _check(load().ipv_init(ctypes.byref(opt)))


def shutdown() -> None:
    load().ipv_shutdown()


def recent_frames(n_frames: int) -> int:
    return load().ipv_recent_frames(n_frames)


def compress(k: KV, v: KV, n_layers: int, n_kv_heads: int, head_dim: int, n_tokens: int,
             frame_grid_h: int, frame_grid_w: int, budget: int, tar_ratio: float,
             kept_idx_out, stream=None) -> None:
    """ipv_compress; flips k.cur and v.cur unless the cache was passed through."""
    _check(load().ipv_compress(ctypes.byref(k), ctypes.byref(v), n_layers, n_kv_heads, head_dim,
                               n_tokens, frame_grid_h, frame_grid_w, budget, tar_ratio,
                               _ptr(kept_idx_out), _stream(stream)))


STATIC_SCRATCH_BYTES = 32 << 20


def compress_static(k: KV, v: KV, dtype: str, token_capacity: int, recent_frames: int,
                    n_layers: int, n_kv_heads: int, head_dim: int, n_tokens: int,
                    frame_grid_h: int, frame_grid_w: int, budget: int, tar_ratio: float,
                    kept_idx_out, stream=None) -> None:
    """ipv_compress_static: the pass with no device allocation and no ipv_init
    (its working memory is a fixed array in the library's device image)."""
    _check(load().ipv_compress_static(ctypes.byref(k), ctypes.byref(v),
                                      IPV_BF16 if dtype == "bf16" else IPV_F32, token_capacity,
                                      recent_frames, n_layers, n_kv_heads, head_dim, n_tokens,
                                      frame_grid_h, frame_grid_w, budget, tar_ratio,
                                      _ptr(kept_idx_out), _stream(stream)))


def score(k: KV, v: KV, n_layers: int, n_kv_heads: int, head_dim: int, n_tokens: int,
          frame_grid_h: int, frame_grid_w: int, tar_out, van_out, stream=None) -> None:
    _check(load().ipv_score(ctypes.byref(k), ctypes.byref(v), n_layers, n_kv_heads, head_dim,
                            n_tokens, frame_grid_h, frame_grid_w, _ptr(tar_out), _ptr(van_out),
                            _stream(stream)))


def select(tar, van, n_slabs: int, n_tokens: int, frame_grid_h: int, frame_grid_w: int,
           budget: int, tar_ratio: float, kept_idx_out, stream=None) -> None:
    _check(load().ipv_select(_ptr(tar), _ptr(van), n_slabs, n_tokens, frame_grid_h, frame_grid_w,
                             budget, tar_ratio, _ptr(kept_idx_out), _stream(stream)))


def van_pool(van, n_layers: int, n_kv_heads: int, n_tokens: int, frame_grid_h: int,
             frame_grid_w: int, cv_tau, pooled_out, pool_size_out=None, patch_id=None,
             frame_id=None, id_stride: int = 0, stream=None) -> None:
    """ipv_van_pool: layer-adaptive pooled VaN of every row (and each layer's pool size)."""
    tau = (ctypes.c_float * 3)(*[float(t) for t in cv_tau])
    _check(load().ipv_van_pool(_ptr(van), _ptr(patch_id), _ptr(frame_id), id_stride, n_layers,
                               n_kv_heads, n_tokens, frame_grid_h, frame_grid_w, tau,
                               _ptr(pooled_out), _ptr(pool_size_out), _stream(stream)))


def append_frames(k: KV, v: KV, k_new, v_new, n_layers: int, n_kv_heads: int, head_dim: int,
                  row0: int, n_new_frames: int, frame_grid_h: int, frame_grid_w: int,
                  first_frame: int = 0, stream=None) -> None:
    """ipv_append_frames: whole new frames behind row0 in every slab of the live halves."""
    _check(load().ipv_append_frames(ctypes.byref(k), ctypes.byref(v), _ptr(k_new), _ptr(v_new),
                                    n_layers, n_kv_heads, head_dim, row0, n_new_frames,
                                    frame_grid_h, frame_grid_w, first_frame, _stream(stream)))


def set_wait_limit(polls: int) -> None:
    """ipv_set_wait_limit: polls before a wait of the fused pass gives up (0: default)."""
    _check(load().ipv_set_wait_limit(int(polls)))


def device_error() -> int:
    """Timeout bits of the fused pass since the last read (waits for the device)."""
    out = ctypes.c_uint32(0)
    _check(load().ipv_device_error(ctypes.byref(out)))
    return out.value


def profile_enable(on: bool) -> None:
    _check(load().ipv_profile_enable(int(bool(on))))


def profile_collect(timeout_ms: int = 60000):
    """{kernel name: (summed ms, launches)} recorded since the last collect."""
    ms = (ctypes.c_double * NUM_KERNELS)()
    n = (ctypes.c_int64 * NUM_KERNELS)()
    _check(load().ipv_profile_collect(ms, n, timeout_ms))
    return {KERNEL_NAMES[i]: (ms[i], n[i]) for i in range(NUM_KERNELS)}
