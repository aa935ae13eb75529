"""CPU oracle for the InfiniPot-V compression pass (arXiv 2506.15745).

TEST INFRASTRUCTURE ONLY: imported by tests/, ``__graft_entry__.smoke()`` and
the cpu_baseline / reference legs of ``bench.py``; never by the product
package. The arithmetic lives in ``ipv_oracle.cpp`` (plain single-threaded
C++, fp64); this module compiles it with g++ and marshals numpy arrays.

Functions mirror the paper's steps:
  scores()  -- TaR (Sec. 3.1, Eq. tar) and VaN (Sec. 3.2) per past token
  select()  -- split-budget selection (Algorithm 1 steps 3-5, Sec. 3.3)
  gather()  -- compaction K~ = K[:, J, :] (Sec. 3.1, Algorithm 2 last step)
  compress()-- the three in sequence (used to time the oracle)
  van_all(), pool_size(), van_pool(), compress_pooled()
            -- layer-adaptive VaN pooling (Sec. 3.2, Algorithm 2) and the pass
               whose VaN stage ranks pooled VaN
  scores_shared(), van_all_shared(), compress_shared()
            -- one index set per layer shared by its KV heads (Sec. 3.1,
               K~ = K[:, I, :]): scores of the concatenated H x D blocks
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ipv_oracle.cpp")
_LIB = os.path.join(_HERE, "liboracle.so")
# A prebuilt library to load instead (the mutation tests point this at a copy
# of the oracle with a planted mistake); never set on the normal path.
_LIB_OVERRIDE = os.environ.get("IPV_ORACLE_LIB_OVERRIDE")
_lib = None


def build_cmd(src: str = _SRC, out: str = _LIB) -> list[str]:
    return ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-o", out, src]


def build(force: bool = False) -> str:
    """Compile liboracle.so next to its source (no-op when up to date)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        subprocess.run(build_cmd(), check=True)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        if _LIB_OVERRIDE:
            lib = ctypes.CDLL(_LIB_OVERRIDE)
        else:
            build()
            lib = ctypes.CDLL(_LIB)
        P, I64, I32, D = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double
        lib.oracle_recent_frames.argtypes = [I64, I32]
        lib.oracle_recent_frames.restype = I32
        lib.oracle_scores.argtypes = [P, P, I32, I64, I64, I32, I64, I32, I32, P, P, P]
        lib.oracle_scores.restype = I32
        lib.oracle_budget_split.argtypes = [I64, I32, I32, I64, D, P]
        lib.oracle_budget_split.restype = I32
        lib.oracle_select.argtypes = [P, P, I64, I64, I32, I32, I64, D, P, P]
        lib.oracle_select.restype = I32
        lib.oracle_gather_rows.argtypes = [P, P, I64, I64, I64, I64, P, I64]
        lib.oracle_gather_rows.restype = I32
        lib.oracle_gather_patch.argtypes = [P, P, I64, I64, I64, I32, P, I64]
        lib.oracle_gather_patch.restype = I32
        lib.oracle_compress.argtypes = [P, P, I32, I64, I64, I32, I64, I32, I32, I64, D,
                                        P, P, P, P, P, I32, P, I32, I32, P, P, P, I32, I32]
        lib.oracle_uniform_select.argtypes = [I64, I64, I32, I64, P]
        lib.oracle_uniform_select.restype = I32
        lib.oracle_frame_mean.argtypes = [P, I64, I64, I64, I32, P, I64]
        lib.oracle_frame_mean.restype = I32
        lib.oracle_scores_shared.argtypes = [P, P, I32, I64, I32, I64, I32, I64, I32, I32, P, P, P]
        lib.oracle_scores_shared.restype = I32
        lib.oracle_van_all_shared.argtypes = [P, I32, I64, I32, I64, I32, I64, P]
        lib.oracle_van_all_shared.restype = I32
        lib.oracle_compress.restype = I32
        lib.oracle_gather_frame.argtypes = [P, P, I64, I64, I64, I32, P, I64]
        lib.oracle_gather_frame.restype = I32
        lib.oracle_van_all.argtypes = [P, I32, I64, I64, I32, I64, P]
        lib.oracle_van_all.restype = I32
        lib.oracle_pool_size.argtypes = [D, P]
        lib.oracle_pool_size.restype = I32
        lib.oracle_van_pool.argtypes = [P, I64, I32, I64, I32, I32, P, P, I64, P, P, P, P]
        lib.oracle_van_pool.restype = I32
        _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _kv_kind(a: np.ndarray) -> int:
    """1 for bf16 bit patterns (stored as uint16), 0 for float32."""
    if a.dtype == np.uint16:
        return 1
    if a.dtype == np.float32:
        return 0
    raise TypeError(f"K/V must be float32 or bf16 bits (uint16), got {a.dtype}")


def recent_frames(n_frames: int, override: int = 0) -> int:
    """r: the override if positive, else max(1, floor(f/8 + 1/2)) (Appendix B.2: r = 0.125 f)."""
    return _load().oracle_recent_frames(int(n_frames), int(override))


def budget_split(n_tokens: int, p: int, r: int, budget: int, alpha: float):
    """(recent kept, TaR picks, VaN picks); None for the pass-through case."""
    out = np.zeros(3, np.int64)
    rc = _load().oracle_budget_split(n_tokens, p, r, budget, float(alpha), _ptr(out))
    if rc != 0:
        raise ValueError("no valid budget split for these arguments")
    return None if out[0] < 0 else tuple(int(x) for x in out)


def scores(k: np.ndarray, v: np.ndarray, n_tokens: int, p: int, r: int,
           patch_id: np.ndarray | None = None):
    """TaR, VaN in fp64 for K, V of shape [S, cap, D] (float32 or bf16 bits)."""
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    assert k.shape == v.shape and k.dtype == v.dtype and k.ndim == 3
    S, cap, D = k.shape
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
        assert patch_id.shape == (S, cap)
    tar = np.empty((S, n_tokens), np.float64)
    van = np.empty((S, n_tokens), np.float64)
    rc = _load().oracle_scores(_ptr(k), _ptr(v), _kv_kind(k), S, cap, D, n_tokens, p, r,
                               _ptr(patch_id), _ptr(tar), _ptr(van))
    if rc != 0:
        raise ValueError("oracle_scores rejected its arguments")
    return tar, van


def select(tar: np.ndarray, van: np.ndarray, n_tokens: int, p: int, r: int, budget: int,
           alpha: float, with_gaps: bool = False):
    """kept indices [S, budget] ascending (and per-stage boundary gaps [S, 2])."""
    tar = np.ascontiguousarray(tar, dtype=np.float64)
    van = np.ascontiguousarray(van, dtype=np.float64)
    S = tar.shape[0]
    assert tar.shape == (S, n_tokens) and van.shape == tar.shape
    kept = np.empty((S, budget), np.int32)
    gaps = np.empty((S, 2), np.float64)
    rc = _load().oracle_select(_ptr(tar), _ptr(van), S, n_tokens, p, r, budget, float(alpha),
                               _ptr(kept), _ptr(gaps))
    if rc != 0:
        raise ValueError("oracle_select rejected its arguments")
    return (kept, gaps) if with_gaps else kept


def gather(src: np.ndarray, kept: np.ndarray, cap_dst: int | None = None,
           dst: np.ndarray | None = None) -> np.ndarray:
    """dst[s, j] = src[s, kept[s, j]] (rows with kept == -1 untouched)."""
    src = np.ascontiguousarray(src)
    kept = np.ascontiguousarray(kept, dtype=np.int32)
    S, cap, D = src.shape
    budget = kept.shape[1]
    cap_dst = cap if cap_dst is None else cap_dst
    if dst is None:
        dst = np.zeros((S, cap_dst, D), src.dtype)
    rc = _load().oracle_gather_rows(_ptr(src), _ptr(dst), D * src.itemsize, S, cap, cap_dst,
                                    _ptr(kept), budget)
    if rc != 0:
        raise ValueError("oracle_gather_rows rejected its arguments")
    return dst


def gather_patch(src_pid: np.ndarray | None, kept: np.ndarray, p: int, cap_src: int,
                 cap_dst: int, dst: np.ndarray | None = None) -> np.ndarray:
    kept = np.ascontiguousarray(kept, dtype=np.int32)
    S, budget = kept.shape
    if dst is None:
        dst = np.zeros((S, cap_dst), np.uint16)
    if src_pid is not None:
        src_pid = np.ascontiguousarray(src_pid, dtype=np.uint16)
    rc = _load().oracle_gather_patch(_ptr(src_pid), _ptr(dst), S, cap_src, cap_dst, p,
                                     _ptr(kept), budget)
    if rc != 0:
        raise ValueError("oracle_gather_patch rejected its arguments")
    return dst


def compress(k: np.ndarray, v: np.ndarray, n_tokens: int, p: int, r: int, budget: int,
             alpha: float, patch_id: np.ndarray | None = None):
    """Whole pass: returns (kept [S,budget], K~ [S,cap,D], V~ [S,cap,D], patch ids [S,cap])."""
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    S, cap, D = k.shape
    kd = np.zeros_like(k)
    vd = np.zeros_like(v)
    pd = np.zeros((S, cap), np.uint16)
    kept = np.empty((S, budget), np.int32)
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
    rc = _load().oracle_compress(_ptr(k), _ptr(v), _kv_kind(k), S, cap, D, n_tokens, p, r,
                                 budget, float(alpha), _ptr(patch_id), _ptr(kd), _ptr(vd),
                                 _ptr(pd), _ptr(kept), 0, None, 1, 0, None, None, None, 0, 0)
    if rc != 0:
        raise ValueError("oracle_compress rejected its arguments")
    return kept, kd, vd, pd


def _tau(tau) -> np.ndarray:
    t = np.ascontiguousarray(tau, dtype=np.float64)
    assert t.shape == (3,)
    return t


def van_all(v: np.ndarray, n_tokens: int) -> np.ndarray:
    """VaN of every row 0..n_tokens-1 (recent frames included), fp64 [S, n_tokens]."""
    v = np.ascontiguousarray(v)
    S, cap, D = v.shape
    out = np.empty((S, n_tokens), np.float64)
    if _load().oracle_van_all(_ptr(v), _kv_kind(v), S, cap, D, n_tokens, _ptr(out)) != 0:
        raise ValueError("oracle_van_all rejected its arguments")
    return out


def pool_size(cv: float, tau) -> int:
    """g(CV) of Algorithm 2 for thresholds tau = (tau_1, tau_2, tau_3)."""
    return _load().oracle_pool_size(float(cv), _ptr(_tau(tau)))


def van_pool(van: np.ndarray, n_kv_heads: int, grid_h: int, grid_w: int, tau,
             patch_id: np.ndarray | None = None, frame_id: np.ndarray | None = None):
    """Layer-adaptive pooled VaN (Sec. 3.2, Algorithm 2) of van [S, N] (every
    cached row). Returns (pooled [S, N], pool size per layer, CV per layer)."""
    van = np.ascontiguousarray(van, dtype=np.float64)
    S, N = van.shape
    stride = N
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
        frame_id = np.ascontiguousarray(frame_id, dtype=np.uint32)
        assert patch_id.shape == frame_id.shape and patch_id.shape[0] == S
        stride = patch_id.shape[1]
    pooled = np.empty_like(van)
    L = S // n_kv_heads
    ks = np.empty(L, np.int32)
    cvs = np.empty(L, np.float64)
    rc = _load().oracle_van_pool(_ptr(van), S, n_kv_heads, N, grid_h, grid_w, _ptr(patch_id),
                                 _ptr(frame_id), stride, _ptr(_tau(tau)), _ptr(pooled),
                                 _ptr(ks), _ptr(cvs))
    if rc != 0:
        raise ValueError("oracle_van_pool rejected its arguments")
    return pooled, ks, cvs


def compress_pooled(k: np.ndarray, v: np.ndarray, n_tokens: int, grid_h: int, grid_w: int,
                    r: int, budget: int, alpha: float, tau, n_kv_heads: int,
                    patch_id: np.ndarray | None = None, frame_id: np.ndarray | None = None):
    """Whole pass whose VaN stage ranks layer-adaptive pooled VaN. Returns
    (kept, K~, V~, patch ids, frame ids, pool size per layer)."""
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    S, cap, D = k.shape
    p = grid_h * grid_w
    kd, vd = np.zeros_like(k), np.zeros_like(v)
    pd = np.zeros((S, cap), np.uint16)
    fd = np.zeros((S, cap), np.uint32)
    kept = np.empty((S, budget), np.int32)
    ks = np.zeros(S // n_kv_heads, np.int32)
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
        frame_id = np.ascontiguousarray(frame_id, dtype=np.uint32)
    rc = _load().oracle_compress(_ptr(k), _ptr(v), _kv_kind(k), S, cap, D, n_tokens, p, r,
                                 budget, float(alpha), _ptr(patch_id), _ptr(kd), _ptr(vd),
                                 _ptr(pd), _ptr(kept), 1, _ptr(_tau(tau)), n_kv_heads,
                                 grid_w, _ptr(frame_id), _ptr(fd), _ptr(ks), 0, 0)
    if rc != 0:
        raise ValueError("oracle_compress rejected its arguments")
    return kept, kd, vd, pd, fd, ks


def scores_shared(k: np.ndarray, v: np.ndarray, n_kv_heads: int, n_tokens: int, p: int, r: int,
                  patch_id: np.ndarray | None = None):
    """TaR, VaN [L, n_tokens] of the concatenated H x D head blocks of each layer."""
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    S, cap, D = k.shape
    L = S // n_kv_heads
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
    tar = np.empty((L, n_tokens), np.float64)
    van = np.empty((L, n_tokens), np.float64)
    rc = _load().oracle_scores_shared(_ptr(k), _ptr(v), _kv_kind(k), L, n_kv_heads, cap, D,
                                      n_tokens, p, r, _ptr(patch_id), _ptr(tar), _ptr(van))
    if rc != 0:
        raise ValueError("oracle_scores_shared rejected its arguments")
    return tar, van


def van_all_shared(v: np.ndarray, n_kv_heads: int, n_tokens: int) -> np.ndarray:
    """Norm of the concatenated H x D value block of every row of every layer."""
    v = np.ascontiguousarray(v)
    S, cap, D = v.shape
    L = S // n_kv_heads
    out = np.empty((L, n_tokens), np.float64)
    if _load().oracle_van_all_shared(_ptr(v), _kv_kind(v), L, n_kv_heads, cap, D, n_tokens,
                                     _ptr(out)) != 0:
        raise ValueError("oracle_van_all_shared rejected its arguments")
    return out


def compress_shared(k: np.ndarray, v: np.ndarray, n_tokens: int, grid_h: int, grid_w: int, r: int,
                    budget: int, alpha: float, n_kv_heads: int, patch_id=None, frame_id=None,
                    tau=None):
    """Whole pass with one index set per layer. Returns (kept [L, budget],
    K~, V~, patch ids, frame ids, pool size per layer); tau given: pooled VaN."""
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    S, cap, D = k.shape
    p = grid_h * grid_w
    L = S // n_kv_heads
    kd, vd = np.zeros_like(k), np.zeros_like(v)
    pd = np.zeros((S, cap), np.uint16)
    fd = np.zeros((S, cap), np.uint32)
    kept = np.empty((L, budget), np.int32)
    ks = np.zeros(L, np.int32)
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
    if frame_id is not None:
        frame_id = np.ascontiguousarray(frame_id, dtype=np.uint32)
    pooled = tau is not None
    rc = _load().oracle_compress(_ptr(k), _ptr(v), _kv_kind(k), S, cap, D, n_tokens, p, r,
                                 budget, float(alpha), _ptr(patch_id), _ptr(kd), _ptr(vd),
                                 _ptr(pd), _ptr(kept), int(pooled),
                                 _ptr(_tau(tau)) if pooled else None, n_kv_heads, grid_w,
                                 _ptr(frame_id), _ptr(fd), _ptr(ks), 1, 0)
    if rc != 0:
        raise ValueError("oracle_compress rejected its arguments")
    return kept, kd, vd, pd, fd, ks


ABLATIONS = {"tar_reverse": 1, "van_reverse": 2, "tar_frame": 3, "uniform": 4}


def uniform_select(n_units: int, n_tokens: int, p: int, budget: int) -> np.ndarray:
    """Uniform Select indices [n_units, budget]: the rows of budget/p whole
    frames at regular intervals, counting back from the newest frame."""
    kept = np.empty((n_units, budget), np.int32)
    if _load().oracle_uniform_select(n_units, n_tokens, p, budget, _ptr(kept)) != 0:
        raise ValueError("oracle_uniform_select rejected its arguments")
    return kept


def frame_mean(tar: np.ndarray, n_past: int, p: int, frame_id: np.ndarray | None = None) -> np.ndarray:
    """Frame-level TaR: each past row's TaR replaced by its frame's mean (copy)."""
    t = np.array(tar, dtype=np.float64, copy=True, order="C")
    U, N = t.shape
    stride = N
    if frame_id is not None:
        frame_id = np.ascontiguousarray(frame_id, dtype=np.uint32)
        stride = frame_id.shape[1]
    if _load().oracle_frame_mean(_ptr(t), U, N, n_past, p, _ptr(frame_id), stride) != 0:
        raise ValueError("oracle_frame_mean rejected its arguments")
    return t


def compress_ablation(k: np.ndarray, v: np.ndarray, n_tokens: int, grid_h: int, grid_w: int, r: int,
                      budget: int, alpha: float, ablation: str, patch_id=None, frame_id=None):
    """Whole per-head pass with an ablation variant ("tar_reverse", "van_reverse",
    "tar_frame", "uniform"). Returns (kept, K~, V~, patch ids, frame ids)."""
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    S, cap, D = k.shape
    p = grid_h * grid_w
    kd, vd = np.zeros_like(k), np.zeros_like(v)
    pd = np.zeros((S, cap), np.uint16)
    fd = np.zeros((S, cap), np.uint32)
    kept = np.empty((S, budget), np.int32)
    if patch_id is not None:
        patch_id = np.ascontiguousarray(patch_id, dtype=np.uint16)
    if frame_id is not None:
        frame_id = np.ascontiguousarray(frame_id, dtype=np.uint32)
    rc = _load().oracle_compress(_ptr(k), _ptr(v), _kv_kind(k), S, cap, D, n_tokens, p, r,
                                 budget, float(alpha), _ptr(patch_id), _ptr(kd), _ptr(vd),
                                 _ptr(pd), _ptr(kept), 0, None, 1, grid_w, _ptr(frame_id),
                                 _ptr(fd), None, 0, ABLATIONS[ablation])
    if rc != 0:
        raise ValueError("oracle_compress rejected its arguments")
    return kept, kd, vd, pd, fd
