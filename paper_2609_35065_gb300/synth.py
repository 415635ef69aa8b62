"""Seeded synthetic workloads for prefix-KV retrieval.

This module only describes shapes and draws random inputs: KV element values,
block tables, matched-prefix lengths and source residency.  It holds none of
the retrieval arithmetic (no slot mapping, no offsets into chunks or planes),
so both the CUDA path and the CPU oracle can be fed from it.

Workload shapes follow TempoKV's evaluation (Sec. 5: Llama-3.1-8B-Instruct and
Qwen2.5-14B-Instruct in BF16; Sec. 5.1: prefix KV retained in complete
256-token chunks, prefix cache ratios 50/75/100%), with KV geometries of the
named model families (layers, KV heads, head dim) and paged blocks of 16
tokens.  Datasets are replaced by synthetic prompt lengths.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

#: bf16 bit pattern written into every paged slot before a retrieval: a NaN
#: payload that round-to-nearest-even conversion of a finite float never yields.
SENTINEL_BF16 = 0x7FA5


@dataclass(frozen=True)
class Geometry:
    layers: int
    kv_heads: int
    head_dim: int
    elem_bytes: int = 2
    block_size: int = 16
    chunk_tokens: int = 256

    @property
    def row_elems(self) -> int:
        """Elements of one token's K (or V) row in one layer: H * D."""
        return self.kv_heads * self.head_dim


@dataclass
class Request:
    prompt_tokens: int
    matched_tokens: int                 # retrieved prefix, a multiple of chunk_tokens
    block_table: np.ndarray             # int32 physical block ids, one per prompt block
    residency: str = "host"             # fast-tier stand-in: "host" (pinned) or "device" (HBM)
    store_tokens: int = 0               # computed suffix stored back into chunks
    shared_prefix_tokens: int = 0       # leading tokens whose KV equals request 0's
    first_token: int = 0                # start of the matched range (a multiple of chunk_tokens)
    store_first: int | None = None      # start of the stored range (default: end of the match)

    @property
    def store_start(self) -> int:
        return self.first_token + self.matched_tokens if self.store_first is None else self.store_first


@dataclass
class Workload:
    name: str
    geom: Geometry
    num_blocks: int
    requests: list[Request]
    dist: str = "normal"                # value distribution: "normal" (0,1) or "uniform" [-1,1)
    seed: int = 0
    notes: dict = field(default_factory=dict)

    @property
    def matched_tokens(self) -> int:
        return sum(r.matched_tokens for r in self.requests)

    def chunk_counts(self, r: Request, tokens: int | None = None) -> list[int]:
        """Token counts of the chunks covering ``tokens`` (default: the matched prefix)."""
        n = r.matched_tokens if tokens is None else tokens
        C = self.geom.chunk_tokens
        return [C] * (n // C) + ([n % C] if n % C else [])


def _perm(n: int, seed: int) -> np.ndarray:
    return np.random.default_rng(seed).permutation(n).astype(np.int32)


def _consecutive_tables(perm: np.ndarray, blocks_each: list[int]) -> list[np.ndarray]:
    out, at = [], 0
    for nb in blocks_each:
        out.append(perm[at:at + nb].copy())
        at += nb
    if at > perm.size:
        raise ValueError("not enough blocks in the paged cache")
    return out


def tiny() -> Workload:
    """2 layers, 4 KV heads, head_dim 64, uniform[-1,1) seed 0, one request whose
    512-token matched prefix is 2 chunks in pinned host memory; 128-block cache
    with a seeded random permutation as block table."""
    g = Geometry(2, 4, 64)
    perm = _perm(128, 0)
    reqs = [Request(512, 512, perm[:32].copy(), "host", store_tokens=512, store_first=0)]
    return Workload("tiny", g, 128, reqs, dist="uniform", seed=0)


def llama8b(requests: int = 16, prompt: int = 4096, hit: float = 0.5, num_blocks: int = 20000) -> Workload:
    """Llama-3-8B-shaped KV (32 layers, 8 KV heads, head_dim 128, 128 KiB/token),
    16 requests of 4096-token prompts at 50% prefix hit, 20,000-block cache with
    seeded random free-block assignment; source in pinned host memory."""
    g = Geometry(32, 8, 128)
    nb_each = -(-prompt // g.block_size)
    tables = _consecutive_tables(_perm(num_blocks, 0), [nb_each] * requests)
    matched = int(prompt * hit) // g.chunk_tokens * g.chunk_tokens
    reqs = [Request(prompt, matched, t, "host") for t in tables]
    name = "llama8b" if (requests, num_blocks) == (16, 20000) else f"llama8b_{requests}req_nb{num_blocks}"
    return Workload(name, g, num_blocks, reqs)


def sweep(ratio: float, requests: int = 32, prompt: int = 8192) -> Workload:
    """8B shape, prefix cache ratio sweep: 32 requests of 8192 tokens whose matched
    prefixes are rounded down to 256-token chunks; each request's source is drawn
    with seed 1 (50% HBM staging buffer, 50% pinned host)."""
    g = Geometry(32, 8, 128)
    nb_each = -(-prompt // g.block_size)
    tables = _consecutive_tables(_perm(20000, 0), [nb_each] * requests)
    matched = int(prompt * ratio) // g.chunk_tokens * g.chunk_tokens
    draws = np.random.default_rng(1).random(requests) < 0.5
    reqs = [Request(prompt, matched, t, "device" if d else "host") for t, d in zip(tables, draws)]
    return Workload(f"sweep{int(round(ratio * 100))}", g, 20000, reqs)


def qwen14b(requests: int = 8, prompt: int = 16384, hit: float = 0.75,
            shared_frac: float = 0.10, num_blocks: int = 8192) -> Workload:
    """14B-shaped KV (48 layers, 8 KV heads, head_dim 128, 192 KiB/token), 8 requests
    of 16,384 tokens at 75% prefix hit; the 4096-token computed suffix is stored back
    into 256-token chunks.  The first 10% of each request's matched blocks are one
    shared physical run (a common prefix, identical KV in every request)."""
    g = Geometry(48, 8, 128)
    B = g.block_size
    nb_each = -(-prompt // B)
    matched = int(prompt * hit) // g.chunk_tokens * g.chunk_tokens
    shared_blocks = int(matched // B * shared_frac)
    perm = _perm(num_blocks, 0)
    tables, at = [], 0
    for r in range(requests):
        if r == 0:
            t = perm[:nb_each].copy()
            at = nb_each
        else:
            fresh = perm[at:at + nb_each - shared_blocks]
            at += nb_each - shared_blocks
            t = np.concatenate([tables[0][:shared_blocks], fresh]).astype(np.int32)
        tables.append(t)
    if at > perm.size:
        raise ValueError("not enough blocks")
    reqs = [Request(prompt, matched, t, "host", store_tokens=prompt - matched,
                    shared_prefix_tokens=shared_blocks * B) for t in tables]
    name = "qwen14b" if (requests, num_blocks) == (8, 8192) else f"qwen14b_{requests}req_nb{num_blocks}"
    return Workload(name, g, num_blocks, reqs, notes={"shared_blocks": shared_blocks})


def llama70b(requests: int = 4, prompt: int = 32768, buffer_frac: float = 1.0) -> Workload:
    """70B-shaped KV (80 layers, 8 KV heads, head_dim 128, 320 KiB/token), 4 requests
    with 32,768-token prefixes fully matched; 8192-block cache.  ``buffer_frac`` sizes
    the pinned fast-tier buffer relative to the batch's matched bytes (refilled
    between passes)."""
    g = Geometry(80, 8, 128)
    nb_each = -(-prompt // g.block_size)
    tables = _consecutive_tables(_perm(8192, 0), [nb_each] * requests)
    reqs = [Request(prompt, prompt, t, "host") for t in tables]
    return Workload("llama70b", g, 8192, reqs, notes={"buffer_frac": buffer_frac})


def custom(L, H, D, B, C, num_blocks, prompts, matched, seed=0, dist="uniform",
           elem_bytes=2, residency="host", firsts=None, store_tokens=None) -> Workload:
    """Small ad-hoc workload for tests: consecutive slices of one seeded permutation.
    ``residency`` is one value or one per request; ``firsts`` the matched-range starts."""
    g = Geometry(L, H, D, elem_bytes, B, C)
    n = len(prompts)
    res = [residency] * n if isinstance(residency, str) else list(residency)
    firsts = [0] * n if firsts is None else list(firsts)
    stores = [0] * n if store_tokens is None else list(store_tokens)
    nb = [-(-p // B) for p in prompts]
    tables = _consecutive_tables(_perm(num_blocks, seed), nb)
    reqs = [Request(p, m, t, rs, store_tokens=st, first_token=f)
            for p, m, t, rs, f, st in zip(prompts, matched, tables, res, firsts, stores)]
    return Workload(f"custom_L{L}H{H}D{D}B{B}C{C}", g, num_blocks, reqs, dist=dist, seed=seed)


# ----------------------------------------------------------------------------
# Values
# ----------------------------------------------------------------------------

def fill_values(out, dist: str, generator) -> None:
    """Fill the torch tensor ``out`` (any 2-byte dtype, any device) with bf16 bit
    patterns of seeded random values: ``normal`` (0,1) or ``uniform`` [-1,1).
    fp32 draws are rounded to bf16 by torch (round to nearest even)."""
    import torch
    flat = out.view(-1)
    step = 1 << 28
    for at in range(0, flat.numel(), step):
        n = min(step, flat.numel() - at)
        if dist == "normal":
            v = torch.randn(n, generator=generator, device=out.device, dtype=torch.float32)
        elif dist == "uniform":
            v = torch.rand(n, generator=generator, device=out.device, dtype=torch.float32) * 2 - 1
        else:
            raise ValueError(dist)
        flat[at:at + n].copy_(v.to(torch.bfloat16).view(flat.dtype))


def sentinel(elem_bytes: int) -> int:
    """Sentinel element for any element size: the bf16 pattern repeated (0xA5 for bytes)."""
    if elem_bytes == 1:
        return 0xA5
    return int.from_bytes(SENTINEL_BF16.to_bytes(2, "little") * (elem_bytes // 2), "little")


def fill_bits(out, generator) -> None:
    """Fill the torch tensor ``out`` with seeded random bits (non-bf16 element sizes)."""
    import torch
    flat = out.view(torch.uint8).view(-1)
    step = 1 << 28
    for at in range(0, flat.numel(), step):
        n = min(step, flat.numel() - at)
        flat[at:at + n].copy_(torch.randint(0, 256, (n,), generator=generator,
                                            device=out.device, dtype=torch.int16).to(torch.uint8))


def fill_values_np(out: np.ndarray, dist: str, seed: int) -> None:
    """CPU-only variant of ``fill_values`` for numpy uint16 buffers (small cases)."""
    import torch
    t = torch.from_numpy(out.view(np.int16).reshape(-1))
    fill_values(t, dist, torch.Generator().manual_seed(seed))
