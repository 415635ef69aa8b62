"""Pins for the fp8 chunk oracle (``oracle/kvs_oracle_fp8.c``): checks against facts
that do not come from the oracle.

* ``pin_e4m3_special_values`` -- the E4M3 special values printed by the OCP OFP8
  specification, revision 1.0 (``tests/golden/ofp8_e4m3_special_values.txt``), with
  and without the sign bit.
* ``pin_e4m3_table``       -- all 256 codes decoded against torch's float8_e4m3fn
  (an independent implementation of the same format).
* ``pin_e4m3_encode``      -- encoding of random binary32 values, every midpoint
  between neighbouring codes and its two binary32 neighbours, against torch's
  round-to-nearest-even conversion (below 464, where torch does not overflow).
* ``pin_e4m3_saturation``  -- magnitudes from 448 up, and infinities, give +-448
  (the specification's saturation mode); NaN gives 0x7F.
* ``pin_e4m3_error_bound`` -- |decode(encode(x)) - x| is at most half a unit in the
  last place: 2^-4 |x| for normal magnitudes, 2^-10 for subnormal ones.
* ``pin_bf16``             -- BF16 rounding against torch's float32 -> bfloat16
  conversion (round to nearest even), ties included.
* ``pin_fp8_fancy``        -- retrieval and store-back written a second way with numpy
  advanced indexing and torch's float8 / bfloat16 conversions, on random small
  geometries (B = 1, ragged chunks, several requests, non-zero first token).
* ``pin_fp8_exact_tags``   -- chunks whose values are E4M3 values times a power of two
  per head, with the head maximum at 448 times that power: retrieval places each
  exactly known value at the slot found by *inverting* the block table, and
  store(retrieve(x)) == x bit for bit (codes and scales).
"""
from __future__ import annotations

import os

import numpy as np
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _torch_decode(codes: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(codes, dtype=np.uint8)).view(torch.float8_e4m3fn).float().numpy()


def _torch_encode(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def _torch_bf16(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def pin_e4m3_special_values(lib):
    with open(os.path.join(GOLDEN, "ofp8_e4m3_special_values.txt")) as f:
        rows = [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]
    assert len(rows) == 7
    for name, code, value in rows:
        c = int(code, 16)
        for sign in (0x00, 0x80):
            got = float(lib.kvs_oracle_e4m3_value(c | sign))
            if value == "nan":
                assert np.isnan(got), (name, sign)
            else:
                want = -float(value) if sign else float(value)
                assert got == want and np.signbit(got) == bool(sign), (name, hex(c | sign), got, want)
                if name != "zero" or not sign:
                    assert lib.kvs_oracle_e4m3_code(want) == c | sign, (name, sign)


def pin_e4m3_table(lib):
    codes = np.arange(256, dtype=np.uint8)
    got = oracle.e4m3_decode(codes, lib)
    want = _torch_decode(codes)
    nan = np.isnan(want)
    assert np.array_equal(np.isnan(got), nan) and nan.sum() == 2
    assert np.array_equal(got[~nan], want[~nan])
    assert np.array_equal(np.signbit(got[~nan]), np.signbit(want[~nan]))
    # codes 0x00..0x7E are strictly increasing in value (the encoder's search relies on it)
    assert np.all(np.diff(got[:0x7F]) > 0)


def _midpoints(lib):
    v = oracle.e4m3_decode(np.arange(0x7F, dtype=np.uint8), lib).astype(np.float64)
    mids = ((v[:-1] + v[1:]) / 2).astype(np.float32)
    assert np.array_equal(mids.astype(np.float64), (v[:-1] + v[1:]) / 2)       # exact in binary32
    up = np.nextafter(mids, np.float32(np.inf))
    down = np.nextafter(mids, np.float32(0))
    return np.concatenate([mids, up, down, -mids, -up, -down])


def pin_e4m3_encode(lib):
    rng = np.random.default_rng(7)
    x = np.concatenate([
        rng.uniform(-463.9, 463.9, 200_000),
        rng.standard_normal(200_000) * np.exp2(rng.integers(-14, 8, 200_000)),
        np.ldexp(rng.uniform(-1, 1, 20_000), -12),
        [0.0, -0.0, 447.9, 448.0, -448.0, 463.99, -463.99],
    ]).astype(np.float32)
    x = np.concatenate([x, _midpoints(lib)])
    x = x[np.abs(x) < 464]
    got = oracle.e4m3_encode(x, lib)
    want = _torch_encode(x)
    bad = np.flatnonzero(got != want)
    assert bad.size == 0, [(float(x[i]), hex(got[i]), hex(want[i])) for i in bad[:5]]


def pin_e4m3_saturation(lib):
    big = np.array([448.0, 449.0, 463.9, 464.0, 480.0, 1e6, 3.4e38, np.inf], dtype=np.float32)
    assert np.all(oracle.e4m3_encode(big, lib) == 0x7E)
    assert np.all(oracle.e4m3_encode(-big, lib) == 0xFE)
    nan = np.array([np.nan, -np.nan], dtype=np.float32)
    assert np.all(oracle.e4m3_encode(nan, lib) == 0x7F)


def pin_e4m3_error_bound(lib):
    rng = np.random.default_rng(8)
    x = (rng.standard_normal(300_000) * np.exp2(rng.integers(-12, 9, 300_000))).astype(np.float32)
    x = x[np.abs(x) <= 448]
    back = oracle.e4m3_decode(oracle.e4m3_encode(x, lib), lib).astype(np.float64)
    err = np.abs(back - x.astype(np.float64))
    normal = np.abs(x) >= 2.0 ** -6
    assert np.all(err[normal] <= 2.0 ** -4 * np.abs(x[normal].astype(np.float64)))
    assert np.all(err[~normal] <= 2.0 ** -10)


def pin_bf16(lib):
    rng = np.random.default_rng(9)
    x = (rng.standard_normal(200_000) * np.exp2(rng.integers(-130, 120, 200_000))).astype(np.float32)
    # exact ties: a bf16 value plus half of its last place, both parities
    b = (rng.integers(0, 0x7F00, 50_000).astype(np.uint32) << 16)
    ties = (b | 0x8000).view(np.float32)
    x = np.concatenate([x, ties, -ties, [0.0, -0.0, np.inf, -np.inf, 3.4e38, -3.4e38]]).astype(np.float32)
    got = oracle.bf16_encode(x, lib)
    assert np.array_equal(got, _torch_bf16(x))
    assert oracle.bf16_encode(np.array([np.nan, -np.nan], np.float32), lib).tolist() == [0x7FFF, 0x7FFF]


# ---- layouts -------------------------------------------------------------------------------

def _fp8_chunk(L, H, D, n, rng, lib, nan_free=True):
    """A random fp8 chunk buffer (scale block + codes), finite codes only by default."""
    hdr = oracle.fp8_scale_bytes(L, H, lib)
    buf = np.zeros(hdr + 2 * L * n * H * D, dtype=np.uint8)
    scales = (rng.uniform(0.5, 4.0, 2 * L * H) * np.exp2(rng.integers(-8, 8, 2 * L * H))).astype(np.float32)
    buf[:2 * L * H * 4] = scales.view(np.uint8)
    codes = rng.integers(0, 256, 2 * L * n * H * D).astype(np.uint8)
    if nan_free:
        codes[(codes & 0x7F) == 0x7F] ^= 0x01
    buf[hdr:] = codes
    return buf


def _slots(first, total, B, table):
    t = np.arange(first, first + total, dtype=np.int64)
    return np.asarray(table, np.int64)[t // B] * B + t % B


def _fancy_retrieve(L, H, D, B, planes, first, chunks, ntok, table, lib):
    hdr = oracle.fp8_scale_bytes(L, H, lib)
    slots = _slots(first, sum(ntok), B, table)
    at = 0
    for c, n in zip(chunks, ntok):
        scales = c[:2 * L * H * 4].view(np.float32).reshape(2 * L, H)
        vals = _torch_decode(c[hdr:]).reshape(2 * L, n, H, D)
        prod = (vals * scales[:, None, :, None]).astype(np.float32)        # binary32 products
        bits = _torch_bf16(prod.reshape(-1)).reshape(2 * L, n, H * D)
        for p in range(2 * L):
            planes[p].reshape(-1, H * D)[slots[at:at + n]] = bits[p]
        at += n


def _fancy_store(L, H, D, B, planes, first, chunks, ntok, table, lib):
    hdr = oracle.fp8_scale_bytes(L, H, lib)
    slots = _slots(first, sum(ntok), B, table)
    at = 0
    for c, n in zip(chunks, ntok):
        rows = np.stack([planes[p].reshape(-1, H, D)[slots[at:at + n]] for p in range(2 * L)])   # [2L][n][H][D]
        x = (rows.astype(np.uint32) << 16).view(np.float32)
        fin = np.where(np.isfinite(x), np.abs(x), np.float32(0))
        amax = fin.max(axis=(1, 3)).astype(np.float32)                                           # [2L][H]
        scale = np.where(amax > 0, amax / np.float32(448), np.float32(1)).astype(np.float32)
        with np.errstate(divide="ignore"):
            inv = np.where(amax > 0, np.float32(448) / amax, np.float32(1)).astype(np.float32)
        q = (x * inv[:, None, :, None]).astype(np.float32)
        q = np.where(np.isnan(q), q, np.clip(q, -448, 448)).astype(np.float32).reshape(-1)
        c[:2 * L * H * 4] = scale.reshape(-1).view(np.uint8)
        c[hdr:] = np.where(np.isnan(q), np.uint8(0x7F), _torch_encode(q))
        at += n


def _random_case(seed):
    rng = np.random.default_rng(seed)
    L, H = int(rng.integers(1, 4)), int(rng.integers(1, 5))
    D = int(rng.choice([16, 32, 64]))
    B = int(rng.choice([1, 4, 16]))
    C = B * int(rng.integers(1, 4))
    reqs, used = [], 0
    for _ in range(int(rng.integers(1, 4))):
        first = C * int(rng.integers(0, 2))
        m = int(rng.integers(1, 3 * C + 1))
        nblk = -(-(first + m) // B)
        reqs.append((first, m, nblk, used))
        used += nblk
    nb = used + int(rng.integers(0, 5))
    perm = rng.permutation(nb).astype(np.int32)
    out = []
    for first, m, nblk, at in reqs:
        ntok = [C] * (m // C) + ([m % C] if m % C else [])
        out.append((first, ntok, perm[at:at + nblk]))
    return rng, L, H, D, B, nb, out


def pin_fp8_fancy(lib):
    for seed in range(20):
        rng, L, H, D, B, nb, reqs = _random_case(seed)
        P, nslot = 2 * L, nb * B
        a = [np.full(nslot * H * D, 0x7FA5, np.uint16) for _ in range(P)]
        b = [x.copy() for x in a]
        stored = []
        for first, ntok, table in reqs:
            chunks = [_fp8_chunk(L, H, D, n, rng, lib) for n in ntok]
            assert oracle.retrieve_fp8(L, H, D, B, a, nb, first, chunks, ntok, table, lib=lib) == 0
            _fancy_retrieve(L, H, D, B, b, first, chunks, ntok, table, lib)
            stored.append((first, ntok, table))
        for p in range(P):
            assert np.array_equal(a[p], b[p]), (seed, p)
        # store-back from the planes just filled, both ways; a few NaN and infinite
        # elements among the stored tokens (excluded from amax, NaN -> 0x7F, inf -> +-448)
        for p in range(P):
            slot_ids = np.concatenate([_slots(f, sum(nt), B, tb) for f, nt, tb in stored])
            pick = rng.choice(slot_ids, size=min(3, slot_ids.size), replace=False)
            for k, sl in enumerate(pick):
                a[p].reshape(-1, H, D)[sl, k % H, (7 * k) % D] = [0x7FC0, 0x7F80, 0xFF80][k % 3]
        for first, ntok, table in stored:
            hdr = oracle.fp8_scale_bytes(L, H, lib)
            ca = [np.zeros(hdr + P * n * H * D, np.uint8) for n in ntok]
            cb = [np.zeros_like(c) for c in ca]
            assert oracle.store_fp8(L, H, D, B, a, nb, first, ca, ntok, table, lib=lib) == 0
            _fancy_store(L, H, D, B, a, first, cb, ntok, table, lib)
            for x, y in zip(ca, cb):
                assert np.array_equal(x, y), seed


def pin_fp8_exact_tags(lib):
    """Per head, values are E4M3 values times 2^k_h with the head's maximum at exactly
    448 * 2^k_h, so scale = 2^k_h, inv = 2^-k_h and every conversion is exact."""
    rng = np.random.default_rng(11)
    for L, H, D, B, first, ntok in [(2, 3, 16, 4, 0, [8, 8, 5]), (1, 2, 32, 1, 8, [8, 3]),
                                    (3, 1, 16, 16, 32, [32, 32])]:
        P = 2 * L
        total = sum(ntok)
        nblk = -(-(first + total) // B)
        nb = nblk + 3
        table = rng.permutation(nb)[:nblk].astype(np.int32)
        hdr = oracle.fp8_scale_bytes(L, H, lib)
        chunks, want = [], {}
        for j, n in enumerate(ntok):
            c = np.zeros(hdr + P * n * H * D, np.uint8)
            k = rng.integers(-6, 6, (P, H))
            scales = np.exp2(k).astype(np.float32)
            c[:P * H * 4] = scales.reshape(-1).view(np.uint8)
            codes = rng.integers(0, 0x7E, (P, n, H, D)).astype(np.uint8) | (rng.integers(0, 2, (P, n, H, D)) << 7).astype(np.uint8)
            codes[:, 0, :, 0] = 0x7E                                 # the head maximum, 448
            c[hdr:] = codes.reshape(-1)
            chunks.append(c)
            s0 = first + sum(ntok[:j])
            for p in range(P):
                for i in range(n):
                    for h in range(H):
                        vals = _torch_decode(codes[p, i, h]) * scales[p, h]
                        want[(p, s0 + i, h)] = _torch_bf16(vals.astype(np.float32))
        planes = [np.full(nb * B * H * D, 0x7FA5, np.uint16) for _ in range(P)]
        assert oracle.retrieve_fp8(L, H, D, B, planes, nb, first, chunks, ntok, table, lib=lib) == 0
        inverse = {int(b): i for i, b in enumerate(table)}
        seen = 0
        for p in range(P):
            rows = planes[p].reshape(nb * B, H, D)
            for slot in range(nb * B):
                blk, off = divmod(slot, B)
                t = inverse[blk] * B + off if blk in inverse else -1
                for h in range(H):
                    if (p, t, h) in want:
                        assert np.array_equal(rows[slot, h], want[(p, t, h)]), (p, t, h)
                        seen += 1
                    else:
                        assert np.all(rows[slot, h] == 0x7FA5), (p, slot, h)
        assert seen == len(want)
        back = [np.zeros_like(c) for c in chunks]
        assert oracle.store_fp8(L, H, D, B, planes, nb, first, back, ntok, table, lib=lib) == 0
        for c, r in zip(chunks, back):
            assert np.array_equal(c, r)


ALL_PINS = [pin_e4m3_special_values, pin_e4m3_table, pin_e4m3_encode, pin_e4m3_saturation,
            pin_e4m3_error_bound, pin_bf16, pin_fp8_fancy, pin_fp8_exact_tags]
