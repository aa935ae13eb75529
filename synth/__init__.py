"""Seeded synthetic inputs for the compression pass (test and bench harness).

A module of its own: it produces the bytes that both the CUDA path and the
CPU oracle consume, and holds none of the compression method's arithmetic.

Recipe (stand-in for the vision-token KV caches of LLaVA-OneVision-7B /
Qwen2-VL-7B on long-video benchmarks, which are not available here):
  * keys: per (slab, patch) an AR(1) chain across frames with unit-variance
    N(0,1) innovations and a stationary start k_0 ~ N(0, I/(1 - rho^2));
    exactly floor(static_frac * p) patches (a seeded permutation, shared by
    all slabs of a stream) are static (rho_static), the rest dynamic;
  * values: unit Gaussian directions times magnitudes exp(sigma_l g), with
    g = beta_l S + sqrt(1 - beta_l^2) z, z ~ N(0,1) per token and S a smooth
    unit-variance field over each frame's grid (four random low-frequency
    cosines per (slab, frame)); sigma_l runs linearly from value_sigma (first
    layer) to value_sigma_last (last layer) and beta_l from value_locality
    down to 0, so early layers have tight, spatially clustered value norms
    and deep layers dispersed, unclustered ones; with the defaults every
    layer has sigma_l = value_sigma and beta_l = 0 (LogNormal(0, sigma));
  * storage: bf16 (round to nearest even) or fp32, layout [slab][cap][D].
Random numbers come from Philox4x32-10 (Salmon et al., SC 2011) with
counter (frame*p + patch, slab, purpose, dim/4) and key (seed, stream), so
the host (numpy) and device (synth.cu) generators draw the same integers;
their floating-point transforms may differ in the last bits.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, replace

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.cu")
_LIB = os.path.join(_HERE, "libipvsynth.so")
_lib = None


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_kv_heads: int
    head_dim: int
    dtype: str              # "bf16" or "f32"
    grid_h: int
    grid_w: int
    n_frames: int           # f: frames held when the cache reaches |M|
    budget: int             # |C|
    tar_ratio: float        # alpha
    static_frac: float = 0.7
    rho_static: float = 0.99
    rho_dynamic: float = 0.3
    value_sigma: float = 0.5
    n_streams: int = 1
    seed: int = 0
    recent_frames: int = 0  # 0: library default
    stream_frames: int = 0  # streaming run: total frames in the stream
    append_frames: int = 0  # streaming run: frames appended per step
    value_sigma_last: float | None = None  # sigma of the last layer (None: value_sigma)
    value_locality: float = 0.0            # beta of the first layer (falls to 0 at the last)
    van_pool: bool = False                 # layer-adaptive VaN pooling in the pass
    cv_tau: tuple = (0.0, 0.0, 0.0)        # CV thresholds of the pool-size map
    head_shared: bool = False              # one index set per layer for all its KV heads
    ablation: str = "none"                 # a variant of the ablation table for the pass

    @property
    def p(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def n_tokens(self) -> int:
        return self.n_frames * self.p

    @property
    def slabs_per_stream(self) -> int:
        return self.n_layers * self.n_kv_heads

    @property
    def n_slabs(self) -> int:
        return self.n_streams * self.slabs_per_stream

    @property
    def is_bf16(self) -> bool:
        return self.dtype == "bf16"

    @property
    def elem_bytes(self) -> int:
        return 2 if self.is_bf16 else 4

    def scaled(self, **kw) -> "Workload":
        return replace(self, **kw)


CONFIGS = {
    # 1 layer x 2 KV heads, D=64 fp32, 8 frames of 4x4 patches -> 48 tokens
    "tiny": Workload("tiny", 1, 2, 64, "f32", 4, 4, 8, 48, 0.5),
    # LLaVA-OneVision-7B shape: 28 x 4 x 128 bf16, 14x14/frame, 48 frames -> 32
    "llava": Workload("llava", 28, 4, 128, "bf16", 14, 14, 48, 6272, 0.5),
    # Qwen2-VL-7B shape: 16x16/frame, 64 frames -> 12288 tokens, alpha 0.3
    "qwen": Workload("qwen", 28, 4, 128, "bf16", 16, 16, 64, 12288, 0.3,
                     static_frac=0.5, rho_dynamic=0.1),
    # 1 h at 1 fps streamed at the LLaVA shape, 16 frames appended per step
    "stream": Workload("stream", 28, 4, 128, "bf16", 14, 14, 48, 6272, 0.5,
                       stream_frames=3600, append_frames=16),
    # 8 independent streams of an 80-layer x 8-KV-head model, 128 frames of 16x16
    "large": Workload("large", 80, 8, 128, "bf16", 16, 16, 128, 24576, 0.5, n_streams=8),
    # the LLaVA shape with layer-adaptive VaN pooling: value spread grows and
    # spatial clustering fades with depth; the CV thresholds split the 28
    # layers over pool sizes 7, 5, 3 and 1
    "llava_pool": Workload("llava_pool", 28, 4, 128, "bf16", 14, 14, 48, 6272, 0.5,
                           value_sigma=0.25, value_sigma_last=1.0, value_locality=0.9,
                           van_pool=True, cv_tau=(0.4, 0.6, 0.9)),
    # the LLaVA shape with one index set per layer shared by its 4 KV heads
    "llava_shared": Workload("llava_shared", 28, 4, 128, "bf16", 14, 14, 48, 6272, 0.5,
                             head_shared=True),
    # the pooled workload streamed like "stream" (frame ids travel with the rows)
    "stream_pool": Workload("stream_pool", 28, 4, 128, "bf16", 14, 14, 48, 6272, 0.5,
                            value_sigma=0.25, value_sigma_last=1.0, value_locality=0.9,
                            van_pool=True, cv_tau=(0.4, 0.6, 0.9),
                            stream_frames=3600, append_frames=16),
}


def value_params(w: Workload):
    """Per-layer (sigma_l, beta_l) as float32 arrays [n_layers], or None when
    every layer uses value_sigma with no spatial field."""
    if w.value_sigma_last is None and w.value_locality == 0.0:
        return None
    L = w.n_layers
    frac = np.arange(L, dtype=np.float64) / max(L - 1, 1)
    last = w.value_sigma if w.value_sigma_last is None else w.value_sigma_last
    sigma = w.value_sigma + (last - w.value_sigma) * frac
    beta = w.value_locality * (1.0 - frac) if L > 1 else np.full(1, w.value_locality)
    return sigma.astype(np.float32), beta.astype(np.float32)


def _frame_field(t: int, s_idx, key, gh: int, gw: int) -> np.ndarray:
    """Smooth unit-variance field [S, gh*gw] of frame t for every slab in s_idx
    (the device generator's frame_field, in float64)."""
    S = s_idx.shape[0]
    w = philox4x32_10((np.uint64(t), s_idx, np.uint64(3), np.uint64(0)), key)
    ph = philox4x32_10((np.uint64(t), s_idx, np.uint64(4), np.uint64(0)), key)
    i = (np.arange(gh * gw) // gw).astype(np.float64)[None, :]
    j = (np.arange(gh * gw) % gw).astype(np.float64)[None, :]
    acc = np.zeros((S, gh * gw))
    for a in range(4):
        wa = np.asarray(w[a]).reshape(S, 1)
        u = (wa % np.uint64(3)).astype(np.float64)
        v = ((wa // np.uint64(3)) % np.uint64(3)).astype(np.float64)
        phi = _unit_open(np.asarray(ph[a]).reshape(S, 1))
        acc += np.sqrt(0.5) * np.cos(2.0 * np.pi * (u * i / gh + v * j / gw + phi))
    return acc


def patch_rho(w: Workload, stream: int = 0) -> np.ndarray:
    """AR(1) coefficient per patch: floor(static_frac p) static patches chosen
    by a permutation seeded with (seed, stream), the rest dynamic."""
    rng = np.random.Generator(np.random.PCG64([w.seed, stream, 0x1D5]))
    perm = rng.permutation(w.p)
    rho = np.full(w.p, w.rho_dynamic, np.float32)
    rho[perm[: int(np.floor(w.static_frac * w.p))]] = w.rho_static
    return rho


# ---------------------------------------------------------------- Philox (host)
_M0, _M1 = np.uint64(0xD2511F53), np.uint64(0xCD9E8D57)
_W0, _W1 = np.uint64(0x9E3779B9), np.uint64(0xBB67AE85)
_MASK = np.uint64(0xFFFFFFFF)


def philox4x32_10(ctr, key):
    """Philox4x32-10 on arrays: ctr = (c0, c1, c2, c3), key = (k0, k1)."""
    c0, c1, c2, c3 = (np.asarray(c, np.uint64) & _MASK for c in ctr)
    k0, k1 = (np.asarray(k, np.uint64) & _MASK for k in key)
    for _ in range(10):
        p0 = _M0 * c0
        p1 = _M1 * c2
        c0, c1, c2, c3 = ((p1 >> np.uint64(32)) ^ c1 ^ k0, p1 & _MASK,
                          (p0 >> np.uint64(32)) ^ c3 ^ k1, p0 & _MASK)
        k0 = (k0 + _W0) & _MASK
        k1 = (k1 + _W1) & _MASK
    return c0, c1, c2, c3


def _unit_open(bits):
    return ((bits >> np.uint64(8)).astype(np.float64) + 0.5) / 16777216.0


def _four_normals(r):
    a, b, c, d = r
    r0 = np.sqrt(-2.0 * np.log(_unit_open(a)))
    r1 = np.sqrt(-2.0 * np.log(_unit_open(c)))
    t0 = 2.0 * np.pi * _unit_open(b)
    t1 = 2.0 * np.pi * _unit_open(d)
    return np.stack([r0 * np.cos(t0), r0 * np.sin(t0), r1 * np.cos(t1), r1 * np.sin(t1)], -1)


def _key(w: Workload, stream: int):
    return np.uint64(w.seed & 0xFFFFFFFF), np.uint64(((w.seed >> 32) + stream) & 0xFFFFFFFF)


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    return ((u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def host_generate(w: Workload, stream: int = 0, n_frames: int | None = None,
                  cap: int | None = None, slabs: int | None = None, slab0: int = 0):
    """K, V as numpy [S, cap, D] (float32, or uint16 bf16 bits) of slabs
    slab0 .. slab0 + S - 1, frames 0..n_frames-1 in rows 0..n_frames*p-1
    (rest zero). For small cases, or for slab ranges of a large one."""
    f = w.n_frames if n_frames is None else n_frames
    S = (w.slabs_per_stream - slab0) if slabs is None else slabs
    p, D = w.p, w.head_dim
    cap = f * p if cap is None else cap
    key = _key(w, stream)
    rho = patch_rho(w, stream).astype(np.float64)
    s_idx = np.arange(slab0, slab0 + S, dtype=np.uint64)[:, None, None]
    q_idx = np.arange(p, dtype=np.uint64)[None, :, None]
    c_idx = np.arange(D // 4, dtype=np.uint64)[None, None, :]
    K = np.zeros((S, cap, D), np.float32)
    V = np.zeros((S, cap, D), np.float32)
    x = np.zeros((S, p, D), np.float64)
    vp = value_params(w)
    vparams = None
    if vp is not None:  # per-slab sigma and beta of the slab's layer
        layer = (np.arange(slab0, slab0 + S) // w.n_kv_heads) % w.n_layers
        vparams = (vp[0][layer].astype(np.float64), vp[1][layer].astype(np.float64))
    for t in range(f):
        tok = np.uint64(t * p) + q_idx
        z = _four_normals(philox4x32_10((tok, s_idx, np.uint64(0), c_idx), key)).reshape(S, p, D)
        if t == 0:
            x = z / np.sqrt(1.0 - rho[None, :, None] ** 2)
        else:
            x = rho[None, :, None] * x + z
        x = x.astype(np.float32).astype(np.float64)  # the chain is carried in fp32
        K[:, t * p:(t + 1) * p] = x
        u = _four_normals(philox4x32_10((tok, s_idx, np.uint64(1), c_idx), key)).reshape(S, p, D)
        zm = _four_normals(philox4x32_10((np.uint64(t * p) + q_idx[..., 0], s_idx[..., 0],
                                          np.uint64(2), np.uint64(0)), key))[..., 0]
        if vparams is None:
            mag = np.exp(w.value_sigma * zm) / np.linalg.norm(u, axis=-1)
        else:
            sig_s, beta_s = vparams
            g = zm
            if np.any(beta_s != 0):
                field = _frame_field(t, s_idx[:, 0, 0], key, w.grid_h, w.grid_w)
                g = np.where(beta_s[:, None] != 0,
                             beta_s[:, None] * field + np.sqrt(1.0 - beta_s[:, None] ** 2) * zm, zm)
            mag = np.exp(sig_s[:, None] * g) / np.linalg.norm(u, axis=-1)
        V[:, t * p:(t + 1) * p] = u * mag[..., None]
    if w.is_bf16:
        return to_bf16_bits(K), to_bf16_bits(V)
    return K, V


# ------------------------------------------------------------ device generator
def build_cmd() -> list[str]:
    return ["nvcc", "-O3", "-std=c++17", "-gencode", "arch=compute_103a,code=sm_103a",
            "-lineinfo", "-Xcompiler", "-fPIC", "-shared", "-o", _LIB, _SRC]


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        subprocess.run(build_cmd(), check=True)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB):
            raise RuntimeError(f"{_LIB} is not built; run __graft_entry__.build()")
        lib = ctypes.CDLL(_LIB)
        P, I64, I32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        lib.synth_fill.argtypes = [P, P, I32, I64, I64, I32, I32, I32, I32, I64, P, P,
                                   ctypes.c_float, ctypes.c_uint64, ctypes.c_uint32, I64,
                                   P, P, I32, I32, I32, P]
        lib.synth_fill.restype = I32
        _lib = lib
    return _lib


class DeviceGenerator:
    """Fills device K/V buffers ([S, cap, D] torch tensors) frame block by
    frame block, keeping each AR(1) chain's last key on the device."""

    def __init__(self, w: Workload, n_slabs: int, stream: int = 0, device=None):
        import torch
        self.w, self.n_slabs, self.stream = w, n_slabs, stream
        dev = torch.device("cuda") if device is None else device
        self.rho = torch.from_numpy(patch_rho(w, stream)).to(dev)
        self.state = torch.zeros((n_slabs, w.p, w.head_dim), dtype=torch.float32, device=dev)
        vp = value_params(w)
        self.layer_sigma = self.layer_beta = None
        if vp is not None:
            self.layer_sigma = torch.from_numpy(vp[0]).to(dev)
            self.layer_beta = torch.from_numpy(vp[1]).to(dev)
        self.next_frame = 0

    def fill(self, k, v, row0: int, n_frames: int, slab_base: int = 0):
        import torch
        assert k.is_cuda and v.is_cuda and k.shape == v.shape and k.shape[0] == self.n_slabs
        S, cap, D = k.shape
        rc = _load().synth_fill(k.data_ptr(), v.data_ptr(), int(self.w.is_bf16), S, cap, D,
                                self.w.p, self.next_frame, n_frames, row0,
                                self.rho.data_ptr(), self.state.data_ptr(),
                                self.w.value_sigma, self.w.seed, self.stream, slab_base,
                                None if self.layer_sigma is None else self.layer_sigma.data_ptr(),
                                None if self.layer_beta is None else self.layer_beta.data_ptr(),
                                self.w.n_layers, self.w.n_kv_heads, self.w.grid_w,
                                torch.cuda.current_stream().cuda_stream)
        if rc != 0:
            raise RuntimeError(f"synth_fill failed with code {rc}")
        self.next_frame += n_frames


def device_generate(w: Workload, k, v, stream: int = 0, n_frames: int | None = None,
                    slab_base: int = 0):
    """Fill frames 0..n_frames-1 of device tensors k, v ([S, cap, D])."""
    g = DeviceGenerator(w, k.shape[0], stream, device=k.device)
    g.fill(k, v, 0, w.n_frames if n_frames is None else n_frames, slab_base)
    return g
