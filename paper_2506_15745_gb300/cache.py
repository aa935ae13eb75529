"""Ping-pong KV cache allocated with PyTorch, in the layout libipv.so expects.

K and V are each [2][n_slabs][capacity][head_dim] (two halves of identical
layout, contiguous, bf16 or fp32); patch ids are [2][n_slabs][capacity]
uint16 bit patterns (held in int16 tensors) and frame ids, when kept,
[2][n_slabs][capacity] uint32 bit patterns (held in int32 tensors). A slab is
one (layer, KV head) of one stream: slab = (stream * n_layers + layer) *
n_kv_heads + head.
"""
from __future__ import annotations

import torch

from . import ipv


class PingPongCache:
    def __init__(self, n_slabs: int, capacity: int, head_dim: int, dtype: str = "bf16",
                 device="cuda", patch_ids: bool = True, frame_ids: bool = False):
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.n_slabs, self.capacity, self.head_dim, self.dtype = n_slabs, capacity, head_dim, dtype
        self.k = torch.empty((2, n_slabs, capacity, head_dim), dtype=tdt, device=device)
        self.v = torch.empty_like(self.k)
        self.pid = (torch.empty((2, n_slabs, capacity), dtype=torch.int16, device=device)
                    if patch_ids else None)
        self.fid = (torch.empty((2, n_slabs, capacity), dtype=torch.int32, device=device)
                    if frame_ids else None)
        self.cur = 0
        self.n_tokens = 0

    # Live (readable) halves.
    @property
    def k_live(self) -> torch.Tensor:
        return self.k[self.cur]

    @property
    def v_live(self) -> torch.Tensor:
        return self.v[self.cur]

    @property
    def pid_live(self):
        return None if self.pid is None else self.pid[self.cur]

    def structs(self, pid_valid: bool = True):
        """(KV, KV) for the C ABI. pid_valid=False passes no source patch or
        frame ids (a fresh cache: patch = row mod p, frame = row div p), while
        still asking the pass to write them for the compacted half."""
        pids, fids = [None, None], [None, None]
        if self.pid is not None:
            pids = [self.pid[0], self.pid[1]]
            if not pid_valid:
                pids[self.cur] = None
        if self.fid is not None:
            fids = [self.fid[0], self.fid[1]]
            if not pid_valid:
                fids[self.cur] = None
        k = ipv.KV.from_tensors((self.k[0], self.k[1]), pids, self.cur, fids)
        v = ipv.KV.from_tensors((self.v[0], self.v[1]), (None, None), self.cur)
        return k, v

    def compress(self, n_layers: int, n_kv_heads: int, grid_h: int, grid_w: int, budget: int,
                 tar_ratio: float, kept_out: torch.Tensor, pid_valid: bool = True, stream=None):
        k, v = self.structs(pid_valid)
        ipv.compress(k, v, n_layers, n_kv_heads, self.head_dim, self.n_tokens, grid_h, grid_w,
                     budget, tar_ratio, kept_out, stream)
        if k.cur != self.cur:
            self.cur = k.cur
            self.n_tokens = budget
