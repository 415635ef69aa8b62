"""Device and pinned-host buffers for a synthetic workload (allocation and seeded fill).

Allocates the paged planes ``[2L][NB*B*H*D]`` on the GPU and the chunk buffers
``[L][2][n][H][D]`` of every request in pinned host memory (the fast-tier
stand-in) or in HBM (a staging copy), fills them from :mod:`.synth`, and builds
the :class:`~.kvs.RequestArg` lists for :func:`~.kvs.kvs_retrieve` and
:func:`~.kvs.kvs_store`.  Like :mod:`.synth`, it computes no slot or offset of
the copy itself.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from . import synth
from .kvs import KVS_SRC_DEVICE, KVS_SRC_HOST_PINNED, ChunkArg, RequestArg

_SLAB = 1 << 27          # elements generated at a time on the generator's device
_DTYPES = {1: torch.uint8, 2: torch.int16, 4: torch.int32, 8: torch.int64}
NP_DTYPES = {1: np.uint8, 2: np.uint16, 4: np.uint32, 8: np.uint64}


def _gen_fill(t: torch.Tensor, dist: str, gen: torch.Generator) -> None:
    if t.element_size() == 2:
        synth.fill_values(t, dist, gen)
    else:
        synth.fill_bits(t, gen)


def _fill(dst: torch.Tensor, gen: torch.Generator, dist: str) -> None:
    """Fill ``dst`` with seeded values drawn on ``gen``'s device (bf16 patterns for
    2-byte elements, random bits otherwise)."""
    gdev = gen.device
    if dst.device.type == gdev.type:
        _gen_fill(dst, dist, gen)
        return
    flat = dst.view(-1)
    for at in range(0, flat.numel(), _SLAB):
        n = min(_SLAB, flat.numel() - at)
        tmp = torch.empty(n, dtype=dst.dtype, device=gdev)
        _gen_fill(tmp, dist, gen)
        flat[at:at + n].copy_(tmp, non_blocking=False)


def plane_seed(seed: int, p: int) -> int:
    return 1_000_003 * (seed + 1) + p


@dataclass
class Buffers:
    workload: synth.Workload
    planes: torch.Tensor | None                    # [2L, NB*B*H*D] elements (bf16 bits for e=2), cuda
    chunks: list[list[torch.Tensor]]               # per request: matched-prefix chunks
    store_chunks: list[list[torch.Tensor]]         # per request: computed-suffix chunks (destinations)
    requests: list[RequestArg]
    store_requests: list[RequestArg]
    host_pool: torch.Tensor | None = None
    device_pool: torch.Tensor | None = None
    store_pool: torch.Tensor | None = None
    plane_init: str = "sentinel"
    notes: dict = field(default_factory=dict)

    _ptrs: tuple = (None, None)                    # (planes base address, plane addresses)

    @property
    def plane_ptrs(self) -> list[int]:
        """Addresses of the 2L planes (rows of one contiguous tensor), computed once per
        planes tensor: a call site that passes them every step pays nothing for it."""
        base = int(self.planes.data_ptr())
        if self._ptrs[0] != base:
            row = self.planes.stride(0) * self.planes.element_size()
            self._ptrs = (base, [base + p * row for p in range(self.planes.shape[0])])
        return self._ptrs[1]

    @property
    def payload_bytes(self) -> int:
        g = self.workload.geom
        return sum(r.matched_tokens for r in self.workload.requests) * 2 * g.layers * g.row_elems * g.elem_bytes

    def initial_plane(self, p: int) -> np.ndarray:
        """Plane p as it was before any copy (host numpy array), regenerated from its seed."""
        w = self.workload
        g = w.geom
        n = w.num_blocks * g.block_size * g.row_elems
        npd = NP_DTYPES[g.elem_bytes]
        if self.plane_init == "sentinel":
            return np.full(n, synth.sentinel(g.elem_bytes), dtype=npd)
        dev = self.planes.device
        tmp = torch.empty(n, dtype=_DTYPES[g.elem_bytes], device=dev)
        gen = torch.Generator(device=dev).manual_seed(plane_seed(w.seed, p))
        _gen_fill(tmp, w.dist, gen)
        return tmp.cpu().numpy().view(npd)


def allocate(w: synth.Workload, device: str = "cuda", store: bool = False,
             store_residency: str = "host", plane_init: str = "sentinel",
             gen_device: str | None = None, with_planes: bool = True) -> Buffers:
    """Allocate and fill every buffer of ``w``.

    ``plane_init`` is ``"sentinel"`` (every element = SENTINEL_BF16) or ``"random"``
    (plane p filled from its own seed, :func:`plane_seed`).  ``store`` also allocates
    destination chunks for each request's ``store_tokens`` suffix, sentinel-filled.
    """
    g = w.geom
    C = g.chunk_tokens
    per_tok = 2 * g.layers * g.row_elems               # elements per token
    gen_device = gen_device or device
    gen = torch.Generator(device=gen_device).manual_seed(w.seed)
    pin = torch.device(device).type == "cuda"

    dt = _DTYPES[g.elem_bytes]
    # the sentinel's bit pattern as a value of the (signed) storage dtype
    sent = int(np.array([synth.sentinel(g.elem_bytes)], dtype=NP_DTYPES[g.elem_bytes])
               .view({1: np.uint8, 2: np.int16, 4: np.int32, 8: np.int64}[g.elem_bytes])[0])
    planes = None
    if with_planes:
        n = w.num_blocks * g.block_size * g.row_elems
        planes = torch.empty((2 * g.layers, n), dtype=dt, device=device)
        if plane_init == "sentinel":
            planes.fill_(sent)
        else:
            for p in range(2 * g.layers):
                pg = torch.Generator(device=device).manual_seed(plane_seed(w.seed, p))
                _gen_fill(planes[p], w.dist, pg)

    host_elems = sum(r.matched_tokens for r in w.requests if r.residency == "host") * per_tok
    dev_elems = sum(r.matched_tokens for r in w.requests if r.residency == "device") * per_tok
    host_pool = torch.empty(host_elems, dtype=dt, pin_memory=pin) if host_elems else None
    device_pool = torch.empty(dev_elems, dtype=dt, device=device) if dev_elems else None

    chunks, requests = [], []
    at = {"host": 0, "device": 0}
    for r in w.requests:
        pool = host_pool if r.residency == "host" else device_pool
        mine = []
        for n in w.chunk_counts(r):
            t = pool[at[r.residency]:at[r.residency] + n * per_tok]
            at[r.residency] += n * per_tok
            _fill(t, gen, w.dist)
            mine.append(t)
        chunks.append(mine)
    # shared prefix: the first shared_prefix_tokens of every request equal request 0's
    for ri, r in enumerate(w.requests):
        if ri == 0 or r.shared_prefix_tokens == 0:
            continue
        for j, (dst, src) in enumerate(zip(chunks[ri], chunks[0])):
            k = min(dst.numel() // per_tok, r.shared_prefix_tokens - j * C)
            if k <= 0:
                break
            n = dst.numel() // per_tok
            dst.view(2 * g.layers, n, g.row_elems)[:, :k].copy_(
                src.view(2 * g.layers, n, g.row_elems)[:, :k])
    for r, mine in zip(w.requests, chunks):
        res = KVS_SRC_HOST_PINNED if r.residency == "host" else KVS_SRC_DEVICE
        requests.append(RequestArg(r.block_table, [ChunkArg(t, t.numel() // per_tok, res) for t in mine],
                                   first_token=r.first_token))

    store_chunks, store_requests, store_pool = [], [], None
    if store:
        total = sum(r.store_tokens for r in w.requests) * per_tok
        if store_residency == "host":
            store_pool = torch.empty(total, dtype=dt, pin_memory=pin)
        else:
            store_pool = torch.empty(total, dtype=dt, device=device)
        store_pool.fill_(sent)
        res = KVS_SRC_HOST_PINNED if store_residency == "host" else KVS_SRC_DEVICE
        off = 0
        for r in w.requests:
            mine = []
            for n in w.chunk_counts(r, r.store_tokens):
                mine.append(store_pool[off:off + n * per_tok])
                off += n * per_tok
            store_chunks.append(mine)
            store_requests.append(RequestArg(r.block_table, [ChunkArg(t, t.numel() // per_tok, res) for t in mine],
                                             first_token=r.store_start if r.store_tokens else 0))
    if torch.device(device).type == "cuda":
        # the fills ran on torch's stream; copies issued next on other streams must see them
        torch.cuda.synchronize()
    return Buffers(w, planes, chunks, store_chunks, requests, store_requests,
                   host_pool, device_pool, store_pool, plane_init)


# ----------------------------------------------------------------------------
# fp8 chunks: [scale block][E4M3 codes]
# ----------------------------------------------------------------------------

def fp8_chunk_bytes(g: synth.Geometry, n: int) -> int:
    """Bytes of an fp8 chunk of n tokens: the 2L*H binary32 scale block padded to a
    multiple of 256 bytes, then [L][2][n][H][D] one-byte codes."""
    scale = (2 * g.layers * g.kv_heads * 4 + 255) // 256 * 256
    return scale + 2 * g.layers * n * g.kv_heads * g.head_dim


@dataclass
class Fp8Buffers:
    workload: synth.Workload
    planes: torch.Tensor | None                    # [2L, NB*B*H*D] BF16 bit patterns (int16), cuda
    chunks: list[list[torch.Tensor]]               # per request: fp8 chunk buffers (uint8)
    store_chunks: list[list[torch.Tensor]]         # per request: fp8 destinations of the stored suffix
    requests: list[RequestArg]
    store_requests: list[RequestArg]
    pools: list = field(default_factory=list)

    plane_ptrs = Buffers.plane_ptrs
    _ptrs: tuple = (None, None)

    @property
    def payload_bytes(self) -> int:
        """Bytes of the retrieved fp8 chunks (scale blocks and codes)."""
        return sum(int(t.numel()) for mine in self.chunks for t in mine)

    def initial_plane(self, p: int) -> np.ndarray:
        g = self.workload.geom
        return np.full(self.workload.num_blocks * g.block_size * g.row_elems, synth.SENTINEL_BF16, dtype=np.uint16)


def _fp8_pool(w, counts, residency, device, pin):
    """One pool holding chunks of the given token counts at 256-byte aligned offsets."""
    sizes = [fp8_chunk_bytes(w.geom, n) for n in counts]
    offs, at = [], 0
    for s in sizes:
        offs.append(at)
        at += (s + 255) // 256 * 256
    if residency == "host":
        pool = torch.zeros(max(at, 1), dtype=torch.uint8, pin_memory=pin)
    else:
        pool = torch.zeros(max(at, 1), dtype=torch.uint8, device=device)
    return pool, [pool[o:o + s] for o, s in zip(offs, sizes)]


def fill_fp8_chunk(t: torch.Tensor, g: synth.Geometry, gen: torch.Generator) -> None:
    """Seeded fp8 chunk content: 2L*H positive binary32 scales in [2^-9, 2^-5) (the
    range amax / 448 takes for KV of unit scale) and uniformly random code bytes (NaN
    codes included, at their natural rate of 2 in 256)."""
    ns = 2 * g.layers * g.kv_heads
    dev = gen.device
    sc = (torch.rand(ns, generator=gen, device=dev, dtype=torch.float32) * 4 + 1) * (2.0 ** -9)
    codes = torch.randint(0, 256, (t.numel() - ((ns * 4 + 255) // 256 * 256),), generator=gen, device=dev,
                          dtype=torch.int16).to(torch.uint8)
    t[:ns * 4].copy_(sc.view(torch.uint8).to(t.device))
    t[(ns * 4 + 255) // 256 * 256:].copy_(codes.to(t.device))


def allocate_fp8(w: synth.Workload, device: str = "cuda", store: bool = False,
                 store_residency: str = "host", with_planes: bool = True) -> Fp8Buffers:
    """Sentinel-filled BF16 planes, seeded fp8 chunks for every request's matched prefix
    (pinned host or HBM, per request), and, with ``store``, zeroed fp8 destinations for
    each request's ``store_tokens`` suffix."""
    g = w.geom
    pin = torch.device(device).type == "cuda"
    gen = torch.Generator(device=device).manual_seed(w.seed)
    planes = None
    if with_planes:
        n = w.num_blocks * g.block_size * g.row_elems
        sent = int(np.array([synth.SENTINEL_BF16], dtype=np.uint16).view(np.int16)[0])
        planes = torch.full((2 * g.layers, n), sent, dtype=torch.int16, device=device)
    pools, requests, views = [], [], {}
    for res in ("host", "device"):
        counts = [n for r in w.requests if r.residency == res for n in w.chunk_counts(r)]
        if counts:
            pool, v = _fp8_pool(w, counts, res, device, pin)
            pools.append(pool)
            views[res] = iter(v)
    chunk_lists = []
    for r in w.requests:
        mine = [next(views[r.residency]) for _ in w.chunk_counts(r)]
        for t in mine:
            fill_fp8_chunk(t, g, gen)
        res = KVS_SRC_HOST_PINNED if r.residency == "host" else KVS_SRC_DEVICE
        requests.append(RequestArg(r.block_table, [ChunkArg(t, n, res) for t, n in zip(mine, w.chunk_counts(r))],
                                   first_token=r.first_token))
        chunk_lists.append(mine)
    store_chunks, store_requests = [], []
    if store:
        counts = [n for r in w.requests for n in w.chunk_counts(r, r.store_tokens)]
        if counts:
            pool, views = _fp8_pool(w, counts, store_residency, device, pin)
            pools.append(pool)
            it = iter(views)
            res = KVS_SRC_HOST_PINNED if store_residency == "host" else KVS_SRC_DEVICE
            for r in w.requests:
                cn = w.chunk_counts(r, r.store_tokens)
                mine = [next(it) for _ in cn]
                store_chunks.append(mine)
                store_requests.append(RequestArg(r.block_table, [ChunkArg(t, n, res) for t, n in zip(mine, cn)],
                                                 first_token=r.store_start if r.store_tokens else 0))
        else:
            store_chunks = [[] for _ in w.requests]
            store_requests = [RequestArg(r.block_table, [], 0) for r in w.requests]
    if torch.device(device).type == "cuda":
        torch.cuda.synchronize()
    return Fp8Buffers(w, planes, chunk_lists, store_chunks, requests, store_requests, pools)
