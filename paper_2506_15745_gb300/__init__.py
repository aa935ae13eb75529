"""GB300 (sm_103a) InfiniPot-V KV-cache compression pass (arXiv 2506.15745).

The pass lives in libipv.so (C ABI in include/ipv.h); `ipv` is its binding,
`cache` allocates ping-pong caches with PyTorch, `shard` partitions
independent slabs over ranks.
"""
from . import ipv  # noqa: F401
from .ipv import IpvError, KV  # noqa: F401
