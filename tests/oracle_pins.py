"""Pins for the CPU oracle: checks against facts that do not come from the oracle.

Each ``pin_*`` takes an oracle library handle (``oracle.load()`` or a mutated
build) and raises ``AssertionError`` when the oracle disagrees with:

* ``pin_footprint``  -- the paper's stated KV footprint (Sec. 2.3, Fig. 1: a
  64k-token Llama-3.1-8B prefix is 8 GiB of BF16 KV): bytes written per token.
* ``pin_tags``       -- coordinate tags: every source element carries its own
  (layer, K/V, token, head, dim); after a retrieval each cache element is
  decoded and checked against its position by *inverting* the block table
  (search, not the forward slot formula).
* ``pin_fancy``      -- a second formulation with numpy advanced indexing, on
  random small geometries (B = 1, ragged chunks, row sizes that are not a
  multiple of 16 bytes, non-zero first token, several requests).
* ``pin_roundtrip``  -- store(retrieve(x)) == x and sentinel preservation.
"""
from __future__ import annotations

import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def read_footprints():
    rows = []
    with open(os.path.join(GOLDEN, "paper_kv_footprint.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            name, L, H, D, e, tokens, nbytes = line.split()
            rows.append((name, int(L), int(H), int(D), int(e), int(tokens), int(nbytes)))
    return rows


def _planes(L, nslots, H, D, dtype, sentinel):
    return [np.full(nslots * H * D, sentinel, dtype=dtype) for _ in range(2 * L)]


def pin_footprint(lib):
    """Bytes the oracle writes per token, scaled to the paper's 64k tokens, equal 8 GiB."""
    for name, L, H, D, e, tokens, nbytes in read_footprints():
        dtype = np.dtype(f"<u{e}")
        B, nb, n = 16, 4, 32
        sent = np.iinfo(dtype).max
        planes = _planes(L, nb * B, H, D, dtype, sent)
        chunk = (np.arange(2 * L * n * H * D, dtype=np.int64) % 1000).astype(dtype)
        bt = np.array([2, 0, 3, 1], dtype=np.int32)
        rc = oracle.retrieve(L, H, D, B, planes, nb, 0, [chunk], bt, lib=lib)
        assert rc == 0, rc
        written = sum(int(np.count_nonzero(p != sent)) for p in planes) * e
        per_token = written // n
        assert written == per_token * n
        assert per_token * tokens == nbytes, (name, per_token, tokens, nbytes)
        # the store direction reads exactly the same number of bytes back
        back = np.full_like(chunk, sent)
        rc = oracle.store(L, H, D, B, planes, nb, 0, [back], bt, lib=lib)
        assert rc == 0, rc
        assert int(np.count_nonzero(back != sent)) * e * tokens // n == nbytes


def _tagged_chunks(L, H, D, counts, first_token, dtype):
    """Chunks whose every element encodes (l, kv, t, h, d) in mixed radix (+1, so 0 is free)."""
    chunks, s = [], first_token
    for n in counts:
        l, kv, i, h, d = np.meshgrid(np.arange(L), np.arange(2), np.arange(n),
                                     np.arange(H), np.arange(D), indexing="ij")
        t = s + i
        tag = ((((l * 2 + kv) * 4096 + t) * H + h) * D + d) + 1
        chunks.append(np.ascontiguousarray(tag.astype(dtype)).reshape(-1))
        s += n
    return chunks


def _decode(tag, H, D):
    v = tag.astype(np.int64) - 1
    d = v % D; v //= D
    h = v % H; v //= H
    t = v % 4096; v //= 4096
    return v // 2, v % 2, t, h, d        # l, kv, t, h, d


def _check_tags(L, H, D, B, nb, planes, requests, sentinel):
    # inverse of each request's block table: physical block -> (request, logical index)
    owner = {}
    for r, (first, counts, bt) in enumerate(requests):
        total = sum(counts)
        lo, hi = first // B, (first + total - 1) // B
        for k in range(lo, hi + 1):
            owner[int(bt[k])] = (r, k)
    for p in range(2 * L):
        cache = planes[p].reshape(nb * B, H, D)
        for slot in range(nb * B):
            row = cache[slot]
            blk, off = divmod(slot, B)
            if blk in owner:
                r, k = owner[blk]
                first, counts, _ = requests[r]
                t = k * B + off
                mapped = first <= t < first + sum(counts)
            else:
                mapped = False
            if not mapped:
                assert np.all(row == sentinel), ("unmapped slot written", p, slot)
                continue
            assert not np.any(row == sentinel), ("mapped slot left unwritten", p, slot)
            l, kv, tt, h, d = _decode(row, H, D)
            assert np.all(2 * l + kv == p), ("wrong plane", p, slot)
            assert np.all(tt == t), ("wrong token", p, slot)
            hh, dd = np.meshgrid(np.arange(H), np.arange(D), indexing="ij")
            assert np.array_equal(h, hh) and np.array_equal(d, dd), ("wrong head/dim", p, slot)


def pin_tags(lib):
    cases = [
        # L, H, D, B, NB, elem dtype, requests as (first_token, chunk token counts)
        (2, 4, 8, 16, 24, np.uint32, [(0, [64, 64]), (0, [32, 16])]),
        (1, 2, 4, 2, 16, np.uint16, [(0, [4, 4, 2])]),
        (3, 1, 3, 1, 40, np.uint32, [(4, [8, 8, 3]), (0, [5])]),
        (2, 3, 5, 4, 32, np.uint32, [(8, [16, 12]), (0, [16])]),
    ]
    rng = np.random.default_rng(7)
    for L, H, D, B, nb, dtype, reqs in cases:
        sent = np.iinfo(dtype).max
        planes = _planes(L, nb * B, H, D, dtype, sent)
        perm = rng.permutation(nb).astype(np.int32)
        requests, at = [], 0
        for first, counts in reqs:
            nblk = -(-(first + sum(counts)) // B)
            bt = perm[at:at + nblk]
            at += nblk
            chunks = _tagged_chunks(L, H, D, counts, first, dtype)
            rc = oracle.retrieve(L, H, D, B, planes, nb, first, chunks, bt, lib=lib)
            assert rc == 0, rc
            requests.append((first, counts, bt))
        _check_tags(L, H, D, B, nb, planes, requests, sent)


def _random_case(rng):
    L = int(rng.integers(1, 4)); H = int(rng.integers(1, 5)); D = int(rng.integers(1, 9))
    B = int(rng.choice([1, 2, 4, 16])); C = B * int(rng.integers(1, 5))
    nreq = int(rng.integers(1, 4))
    reqs, nblocks_needed = [], 0
    for _ in range(nreq):
        first = C * int(rng.integers(0, 2))
        nfull = int(rng.integers(0, 3))
        tail = int(rng.integers(0, C))
        counts = [C] * nfull + ([tail] if tail else [])
        reqs.append((first, counts))
        nblocks_needed += -(-(first + sum(counts)) // B) if (first + sum(counts)) else 0
    nb = nblocks_needed + int(rng.integers(0, 6))
    return L, H, D, B, max(nb, 1), reqs


def pin_fancy(lib, cases: int = 40):
    rng = np.random.default_rng(12345)
    for _ in range(cases):
        L, H, D, B, nb, reqs = _random_case(rng)
        dtype = np.dtype(rng.choice(["<u1", "<u2", "<u4"]))
        sent = np.iinfo(dtype).max
        a = _planes(L, nb * B, H, D, dtype, sent)
        b = [p.copy() for p in a]
        perm = rng.permutation(nb).astype(np.int32)
        at = 0
        for first, counts in reqs:
            nblk = -(-(first + sum(counts)) // B)
            bt = perm[at:at + nblk]
            at += nblk
            chunks = [rng.integers(0, sent, size=2 * L * n * H * D, dtype=dtype) for n in counts]
            assert oracle.retrieve(L, H, D, B, a, nb, first, chunks, bt, lib=lib) == 0
            oracle.retrieve_fancy(L, H, D, B, b, first, chunks, bt)
            for pa, pb in zip(a, b):
                assert np.array_equal(pa, pb), ("retrieve differs from fancy indexing", L, H, D, B)
            got = [np.full_like(c, sent) for c in chunks]
            want = [np.full_like(c, sent) for c in chunks]
            assert oracle.store(L, H, D, B, a, nb, first, got, bt, lib=lib) == 0
            oracle.store_fancy(L, H, D, B, b, first, want, bt)
            for ga, wb in zip(got, want):
                assert np.array_equal(ga, wb), ("store differs from fancy indexing", L, H, D, B)


def pin_roundtrip(lib):
    rng = np.random.default_rng(99)
    L, H, D, B, nb = 2, 4, 64, 16, 128
    sent = 0x7FA5
    planes = _planes(L, nb * B, H, D, np.uint16, sent)
    bt = rng.permutation(nb).astype(np.int32)[:32]
    chunks = [rng.integers(0, 0x7F80, size=2 * L * 256 * H * D, dtype=np.uint16) for _ in range(2)]
    assert oracle.retrieve(L, H, D, B, planes, nb, 0, chunks, bt, lib=lib) == 0
    back = [np.zeros_like(c) for c in chunks]
    assert oracle.store(L, H, D, B, planes, nb, 0, back, bt, lib=lib) == 0
    for c, r in zip(chunks, back):
        assert np.array_equal(c, r), "store(retrieve(x)) != x"
    used = set(int(x) for x in bt)
    for p in planes:
        rows = p.reshape(nb, B * H * D)
        for blk in range(nb):
            if blk not in used:
                assert np.all(rows[blk] == sent), "unused block touched"


ALL_PINS = (pin_footprint, pin_tags, pin_fancy, pin_roundtrip)
