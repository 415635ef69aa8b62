"""Element-by-element comparison of GPU results with the CPU oracle.

Expected planes are built on the host from the same seeded inputs the GPU got
(initial plane content + the oracle's retrieval of every request, one plane at
a time so that tens-of-GB caches fit), then compared with the GPU plane copied
back.  Nothing the GPU produced is ever fed to the oracle.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

import oracle
from paper_2609_35065_gb300 import synth
from paper_2609_35065_gb300.buffers import NP_DTYPES

THREADS = min(8, os.cpu_count() or 1)


def host_chunks(buf, which="chunks"):
    """Host numpy views (copies for device chunks) of every request's chunk buffers."""
    npd = NP_DTYPES[buf.workload.geom.elem_bytes]
    out = []
    for mine in getattr(buf, which):
        out.append([(t.numpy() if t.device.type == "cpu" else t.cpu().numpy()).view(npd) for t in mine])
    return out


def expected_plane(buf, p, chunks_np):
    w = buf.workload
    g = w.geom
    exp = buf.initial_plane(p)
    planes = [None] * (2 * g.layers)
    planes[p] = exp
    for r, req in enumerate(w.requests):
        if not chunks_np[r]:
            continue
        rc = oracle.retrieve(g.layers, g.kv_heads, g.head_dim, g.block_size, planes, w.num_blocks,
                             req.first_token, chunks_np[r], req.block_table, p0=p, p1=p + 1)
        assert rc == 0, rc
    return exp


def _diff(got, exp, label):
    if np.array_equal(got, exp):
        return None
    idx = np.flatnonzero(got != exp)
    return f"{label}: {idx.size} elements differ, first at {int(idx[0])} (got {got[idx[0]]:#x}, want {exp[idx[0]]:#x})"


def check_retrieve(buf, planes=None, chunks_np=None):
    """Every element of the listed planes (default: all) equals the oracle's result."""
    g = buf.workload.geom
    npd = NP_DTYPES[g.elem_bytes]
    chunks_np = host_chunks(buf) if chunks_np is None else chunks_np
    planes = range(2 * g.layers) if planes is None else planes

    def one(p):
        got = buf.planes[p].cpu().numpy().view(npd)
        return _diff(got, expected_plane(buf, p, chunks_np), f"plane {p}")

    with ThreadPoolExecutor(THREADS) as ex:
        bad = [x for x in ex.map(one, planes) if x]
    assert not bad, "\n".join(bad[:8])


def check_store(buf, chunks_np=None):
    """The GPU's store-back output equals the oracle's store from the oracle's planes."""
    w = buf.workload
    g = w.geom
    npd = NP_DTYPES[g.elem_bytes]
    chunks_np = host_chunks(buf) if chunks_np is None else chunks_np
    fill = synth.sentinel(g.elem_bytes)
    want = [[np.full(t.numel(), fill, dtype=npd) for t in mine] for mine in buf.store_chunks]

    def one(p):
        exp = expected_plane(buf, p, chunks_np)
        planes = [None] * (2 * g.layers)
        planes[p] = exp
        for r, req in enumerate(buf.store_requests):
            if not want[r]:
                continue
            rc = oracle.store(g.layers, g.kv_heads, g.head_dim, g.block_size, planes, w.num_blocks,
                              req.first_token, want[r], req.block_table, p0=p, p1=p + 1)
            assert rc == 0, rc

    with ThreadPoolExecutor(THREADS) as ex:
        list(ex.map(one, range(2 * g.layers)))
    bad = []
    for r, (mine, exp) in enumerate(zip(buf.store_chunks, want)):
        for j, (t, e) in enumerate(zip(mine, exp)):
            got = (t.numpy() if t.device.type == "cpu" else t.cpu().numpy()).view(npd)
            d = _diff(got, e, f"store request {r} chunk {j}")
            if d:
                bad.append(d)
    assert not bad, "\n".join(bad[:8])


def free(buf):
    for name in ("planes", "host_pool", "device_pool", "store_pool"):
        setattr(buf, name, None)
    buf.chunks = buf.store_chunks = []
    buf.requests = buf.store_requests = []
    torch.cuda.empty_cache()


def random_workload(seed):
    """Small seeded workload of random geometry: 1/2/4/8-byte elements, B in {1..32},
    rows that are not a multiple of 16 bytes, ragged last chunks, non-zero first tokens,
    mixed residency, and a stored suffix on some requests."""
    rng = np.random.default_rng(seed)
    e = int(rng.choice([1, 2, 2, 2, 4, 8]))
    L = int(rng.integers(1, 5))
    H = int(rng.integers(1, 9))
    D = int(rng.choice([1, 3, 5, 8, 64, 128]))
    B = int(rng.choice([1, 2, 8, 16, 32]))
    C = B * int(rng.integers(1, 5))
    nreq = int(rng.integers(1, 5))
    prompts, matched, firsts, res, stores = [], [], [], [], []
    for _ in range(nreq):
        first = C * int(rng.integers(0, 2))
        st = int(rng.integers(0, 2 * C + 1)) if rng.random() < 0.6 else 0
        # a stored suffix starts where the match ends, so that end must be chunk-aligned
        m = C * int(rng.integers(0, 5)) if st else int(rng.integers(0, 4 * C + 1))
        prompts.append(first + m + st + int(rng.integers(0, B + 1)))
        matched.append(m)
        firsts.append(first)
        res.append("device" if rng.random() < 0.4 else "host")
        stores.append(st)
    nb = sum(-(-p // B) for p in prompts) + int(rng.integers(0, 8))
    return synth.custom(L, H, D, B, C, nb, prompts, matched, seed=seed, elem_bytes=e,
                        residency=res, firsts=firsts, store_tokens=stores)


def shared_workload(differ: bool):
    """Three requests whose first two logical blocks name the same two physical blocks
    (a shared prefix); with ``differ`` one token of the third request's copy differs."""
    from paper_2609_35065_gb300 import buffers
    g = synth.Geometry(2, 2, 8, 2, 4, 8)
    perm = np.arange(40, dtype=np.int32)[::-1].copy()
    t0 = perm[:6]
    t1 = np.concatenate([t0[:2], perm[6:10]]).astype(np.int32)
    t2 = np.concatenate([t0[:2], perm[10:12]]).astype(np.int32)
    reqs = [synth.Request(24, 24, t0, "host", shared_prefix_tokens=0),
            synth.Request(24, 24, t1, "device", shared_prefix_tokens=8),
            synth.Request(16, 12, t2, "host", shared_prefix_tokens=8)]
    w = synth.Workload("shared", g, 40, reqs, dist="uniform", seed=3)
    buf = buffers.allocate(w)
    if differ:
        buf.chunks[2][0].view(4, 8, 16)[:, 1, :] += 1          # token 1 of request 2 differs
    return buf


# ---- fp8 chunks ------------------------------------------------------------------

def _np(t):
    return t.numpy() if t.device.type == "cpu" else t.cpu().numpy()


def expected_plane_fp8(buf, p, chunks_np):
    w = buf.workload
    g = w.geom
    exp = buf.initial_plane(p)
    planes = [None] * (2 * g.layers)
    planes[p] = exp
    for r, req in enumerate(w.requests):
        if not chunks_np[r]:
            continue
        ntok = w.chunk_counts(req)
        rc = oracle.retrieve_fp8(g.layers, g.kv_heads, g.head_dim, g.block_size, planes, w.num_blocks,
                                 req.first_token, chunks_np[r], ntok, req.block_table, p0=p, p1=p + 1)
        assert rc == 0, rc
    return exp


def check_retrieve_fp8(buf, chunks_np=None, planes=None):
    """Every element of the BF16 planes equals the oracle's dequantising retrieval."""
    g = buf.workload.geom
    chunks_np = [[_np(t) for t in mine] for mine in buf.chunks] if chunks_np is None else chunks_np
    planes = range(2 * g.layers) if planes is None else planes

    def one(p):
        got = buf.planes[p].cpu().numpy().view(np.uint16)
        return _diff(got, expected_plane_fp8(buf, p, chunks_np), f"plane {p}")

    with ThreadPoolExecutor(THREADS) as ex:
        bad = [x for x in ex.map(one, planes) if x]
    assert not bad, "\n".join(bad[:8])


def check_store_fp8(buf, plane_source="gpu"):
    """The fp8 chunks the GPU stored equal the oracle's quantising store, byte for byte
    (scale blocks and codes), from the planes the GPU read: ``plane_source`` "gpu" reads
    them back (they are the store's input, which the store does not modify), "oracle"
    rebuilds them from the retrieval's oracle."""
    w = buf.workload
    g = w.geom
    want = [[np.zeros(t.numel(), np.uint8) for t in mine] for mine in buf.store_chunks]
    chunks_np = [[_np(t) for t in mine] for mine in buf.chunks]

    def one(p):
        if plane_source == "gpu":
            src = buf.planes[p].cpu().numpy().view(np.uint16)
        else:
            src = expected_plane_fp8(buf, p, chunks_np)
        planes = [None] * (2 * g.layers)
        planes[p] = src
        for r, req in enumerate(buf.store_requests):
            if not want[r]:
                continue
            ntok = [c.num_tokens for c in req.chunks]
            rc = oracle.store_fp8(g.layers, g.kv_heads, g.head_dim, g.block_size, planes, w.num_blocks,
                                  req.first_token, want[r], ntok, req.block_table, p0=p, p1=p + 1)
            assert rc == 0, rc

    with ThreadPoolExecutor(THREADS) as ex:
        list(ex.map(one, range(2 * g.layers)))
    bad = []
    for r, (mine, exp) in enumerate(zip(buf.store_chunks, want)):
        for j, (t, e) in enumerate(zip(mine, exp)):
            d = _diff(_np(t), e, f"fp8 store request {r} chunk {j}")
            if d:
                bad.append(d)
    assert not bad, "\n".join(bad[:8])


def random_fp8_workload(seed):
    """Small seeded workload for fp8 chunks: head_dim a multiple of 16, B in {1..32},
    ragged last chunks, non-zero first tokens, mixed residency, stored suffixes."""
    rng = np.random.default_rng(1000 + seed)
    L = int(rng.integers(1, 4))
    H = int(rng.integers(1, 9))
    D = int(rng.choice([16, 32, 64, 128]))
    B = int(rng.choice([1, 2, 8, 16, 32]))
    C = B * int(rng.integers(1, 5))
    nreq = int(rng.integers(1, 4))
    prompts, matched, firsts, res, stores = [], [], [], [], []
    for _ in range(nreq):
        first = C * int(rng.integers(0, 2))
        st = int(rng.integers(0, 2 * C + 1)) if rng.random() < 0.6 else 0
        m = C * int(rng.integers(0, 5)) if st else int(rng.integers(0, 4 * C + 1))
        prompts.append(first + m + st + int(rng.integers(0, B + 1)))
        matched.append(m)
        firsts.append(first)
        res.append("device" if rng.random() < 0.4 else "host")
        stores.append(st)
    nb = sum(-(-p // B) for p in prompts) + int(rng.integers(0, 8))
    return synth.custom(L, H, D, B, C, nb, prompts, matched, seed=seed, residency=res, firsts=firsts,
                        store_tokens=stores)
