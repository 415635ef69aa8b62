"""CPU oracle for prefix-KV retrieval and store-back (TempoKV, Sec. 2.1, 4, 5.1).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA path and never imports it.

Two independent formulations of the same definition (see ``kvs_oracle.c``):

* ``retrieve`` / ``store``: the C element loop in ``kvs_oracle.c`` (the oracle
  proper), called through ctypes on numpy arrays.
* ``retrieve_fancy`` / ``store_fancy``: the same assignment written with numpy
  advanced indexing (a library routine), used to pin the C loop.

Layouts (TempoKV reuses the LMCache/vLLM transfer path, Sec. 4): a chunk of
``n`` tokens is ``[L][2][n][H][D]``; a paged plane ``p = 2*l + kv`` is
``[NB*B][H][D]``; request token ``t`` lives in slot
``block_table[t // B] * B + t % B``.  Prefix KV is retained in complete
256-token chunks (Sec. 5.1, Workload), in BF16 (Sec. 5, setup); elements are
copied as opaque ``e``-byte values.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvs_oracle.c")
_SRC_FP8 = os.path.join(_HERE, "kvs_oracle_fp8.c")
_SO = os.path.join(_HERE, "_build", "libkvs_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``kvs_oracle.c`` and ``kvs_oracle_fp8.c`` with gcc into ``oracle/_build``
    (plain -O2, no tuning; ISO C, so binary32 expressions are evaluated as written,
    each operation rounded once, with no fused multiply-add)."""
    os.makedirs(os.path.dirname(_SO), exist_ok=True)
    srcs = [_SRC, _SRC_FP8]
    if force or not os.path.exists(_SO) or any(os.path.getmtime(_SO) < os.path.getmtime(x) for x in srcs):
        tmp = _SO + f".{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-shared", "-fPIC", *srcs,
                        "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _SO)
    return _SO


def load(path: str | None = None):
    """Load (building first if needed) the oracle library; ``path`` loads another build."""
    global _lib
    if path is not None:
        return _bind(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
    return _lib


def _bind(lib):
    P = ctypes.c_void_p
    sig = [ctypes.c_int] * 5 + [P, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
                                ctypes.c_int64, ctypes.c_int, P, P, P, ctypes.c_int64]
    for name in ("kvs_oracle_retrieve", "kvs_oracle_store"):
        fn = getattr(lib, name)
        fn.argtypes = sig
        fn.restype = ctypes.c_int
    lib.kvs_oracle_fill.argtypes = [P, ctypes.c_int64, ctypes.c_int, P]
    lib.kvs_oracle_fill.restype = None
    sig8 = [ctypes.c_int] * 4 + [P, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
                                 ctypes.c_int64, ctypes.c_int, P, P, P, ctypes.c_int64]
    for name in ("kvs_oracle_retrieve_fp8", "kvs_oracle_store_fp8"):
        fn = getattr(lib, name)
        fn.argtypes = sig8
        fn.restype = ctypes.c_int
    lib.kvs_oracle_e4m3_value.argtypes = [ctypes.c_uint8]
    lib.kvs_oracle_e4m3_value.restype = ctypes.c_float
    lib.kvs_oracle_e4m3_code.argtypes = [ctypes.c_float]
    lib.kvs_oracle_e4m3_code.restype = ctypes.c_uint8
    lib.kvs_oracle_bf16_bits.argtypes = [ctypes.c_float]
    lib.kvs_oracle_bf16_bits.restype = ctypes.c_uint16
    lib.kvs_oracle_fp8_scale_bytes.argtypes = [ctypes.c_int, ctypes.c_int]
    lib.kvs_oracle_fp8_scale_bytes.restype = ctypes.c_int64
    for name in ("kvs_oracle_e4m3_encode_array", "kvs_oracle_e4m3_decode_array", "kvs_oracle_bf16_encode_array"):
        fn = getattr(lib, name)
        fn.argtypes = [P, P, ctypes.c_int64]
        fn.restype = None
    return lib


def _ptr(a: np.ndarray | None) -> int:
    if a is None:
        return 0
    if not a.flags.c_contiguous:
        raise ValueError("oracle buffers must be C-contiguous")
    return a.ctypes.data


def _call(name, L, H, D, B, planes, num_blocks, first_token, chunks, block_table, p0, p1, lib):
    lib = lib or load()
    e = None
    for a in list(planes) + list(chunks):
        if a is not None:
            e = a.dtype.itemsize
            break
    if e is None:
        raise ValueError("no buffers")
    p1 = 2 * L if p1 is None else p1
    plane_ptrs = (ctypes.c_void_p * (2 * L))(*[_ptr(a) for a in planes])
    chunk_ptrs = (ctypes.c_void_p * max(1, len(chunks)))(*[_ptr(c) for c in chunks])
    ntok = (ctypes.c_int32 * max(1, len(chunks)))(*[_chunk_tokens(c, L, H, D) for c in chunks])
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    rc = getattr(lib, name)(L, H, D, e, B, plane_ptrs, int(num_blocks), p0, p1,
                            int(first_token), len(chunks), chunk_ptrs, ntok,
                            bt.ctypes.data, bt.size)
    return rc


def _chunk_tokens(chunk: np.ndarray, L: int, H: int, D: int) -> int:
    per_token = 2 * L * H * D
    if chunk.size % per_token:
        raise ValueError(f"chunk of {chunk.size} elements is not a whole number of tokens")
    return chunk.size // per_token


def retrieve(L, H, D, B, planes, num_blocks, first_token, chunks, block_table,
             p0=0, p1=None, lib=None) -> int:
    """Scatter one request's chunks into ``planes`` (list of 2L arrays, [NB*B*H*D] each).

    Returns the C oracle's status: 0, or -2 when a token has no valid block.
    """
    return _call("kvs_oracle_retrieve", L, H, D, B, planes, num_blocks, first_token,
                 chunks, block_table, p0, p1, lib)


def store(L, H, D, B, planes, num_blocks, first_token, chunks, block_table,
          p0=0, p1=None, lib=None) -> int:
    """Gather one request's tokens from ``planes`` into its chunk buffers (in place)."""
    return _call("kvs_oracle_store", L, H, D, B, planes, num_blocks, first_token,
                 chunks, block_table, p0, p1, lib)


def fill(a: np.ndarray, value: int) -> None:
    """Fill ``a`` with the element bit pattern ``value`` (little-endian), via the C loop."""
    e = a.dtype.itemsize
    pat = np.array([value], dtype=f"<u{e}").view(np.uint8)
    load().kvs_oracle_fill(_ptr(a), a.size, e, pat.ctypes.data)


# ----------------------------------------------------------------------------
# Second formulation: numpy advanced indexing (library routine special case).
# ----------------------------------------------------------------------------

def _slots_fancy(first_token, total_tokens, B, block_table):
    t = np.arange(first_token, first_token + total_tokens, dtype=np.int64)
    bt = np.asarray(block_table, dtype=np.int64)
    return bt[t // B] * B + t % B


def retrieve_fancy(L, H, D, B, planes, first_token, chunks, block_table):
    """Same assignment as ``retrieve`` with numpy fancy indexing; planes must be valid."""
    if not chunks:
        return
    per_chunk = [c.reshape(L, 2, -1, H * D) for c in chunks]
    rows = np.concatenate(per_chunk, axis=2)               # [L][2][T][H*D]
    slots = _slots_fancy(first_token, rows.shape[2], B, block_table)
    for l in range(L):
        for kv in range(2):
            planes[2 * l + kv].reshape(-1, H * D)[slots] = rows[l, kv]


def store_fancy(L, H, D, B, planes, first_token, chunks, block_table):
    """Same assignment as ``store`` with numpy fancy indexing; writes into ``chunks``."""
    if not chunks:
        return
    ntok = [c.size // (2 * L * H * D) for c in chunks]
    slots = _slots_fancy(first_token, sum(ntok), B, block_table)
    start = 0
    for c, n in zip(chunks, ntok):
        view = c.reshape(L, 2, n, H * D)
        for l in range(L):
            for kv in range(2):
                view[l, kv] = planes[2 * l + kv].reshape(-1, H * D)[slots[start:start + n]]
        start += n


# ----------------------------------------------------------------------------
# fp8 chunks (kvs_oracle_fp8.c): E4M3 codes of the OCP OFP8 specification,
# revision 1.0, with one binary32 scale per (chunk, layer, K/V, head).
# ----------------------------------------------------------------------------

def fp8_scale_bytes(L: int, H: int, lib=None) -> int:
    """Bytes of the scale block at the head of an fp8 chunk buffer."""
    return int((lib or load()).kvs_oracle_fp8_scale_bytes(L, H))


def fp8_chunk_bytes(L: int, H: int, D: int, n: int, lib=None) -> int:
    """Bytes of an fp8 chunk buffer of n tokens: scale block + [L][2][n][H][D] codes."""
    return fp8_scale_bytes(L, H, lib) + 2 * L * n * H * D


def e4m3_encode(x: np.ndarray, lib=None) -> np.ndarray:
    """E4M3 codes of float32 values (round to nearest even, saturating; NaN -> 0x7F)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint8)
    (lib or load()).kvs_oracle_e4m3_encode_array(_ptr(x), _ptr(out), x.size)
    return out


def e4m3_decode(c: np.ndarray, lib=None) -> np.ndarray:
    """float32 values of E4M3 codes (NaN for 0x7F / 0xFF)."""
    c = np.ascontiguousarray(c, dtype=np.uint8)
    out = np.empty(c.shape, dtype=np.float32)
    (lib or load()).kvs_oracle_e4m3_decode_array(_ptr(c), _ptr(out), c.size)
    return out


def bf16_encode(x: np.ndarray, lib=None) -> np.ndarray:
    """BF16 bit patterns of float32 values (round to nearest even; NaN -> 0x7FFF)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    (lib or load()).kvs_oracle_bf16_encode_array(_ptr(x), _ptr(out), x.size)
    return out


def _call_fp8(name, L, H, D, B, planes, num_blocks, first_token, chunks, chunk_tokens, block_table,
              p0, p1, lib):
    lib = lib or load()
    p1 = 2 * L if p1 is None else p1
    for a in planes:
        if a is not None and a.dtype != np.uint16:
            raise ValueError("fp8 oracle planes hold BF16 bit patterns (uint16)")
    for c in chunks:
        if c.dtype != np.uint8:
            raise ValueError("fp8 chunks are byte buffers (uint8)")
    plane_ptrs = (ctypes.c_void_p * (2 * L))(*[_ptr(a) for a in planes])
    chunk_ptrs = (ctypes.c_void_p * max(1, len(chunks)))(*[_ptr(c) for c in chunks])
    ntok = (ctypes.c_int32 * max(1, len(chunks)))(*[int(n) for n in chunk_tokens])
    for c, n in zip(chunks, chunk_tokens):
        if c.size < fp8_chunk_bytes(L, H, D, n, lib):
            raise ValueError("fp8 chunk buffer smaller than its scale block and codes")
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    return getattr(lib, name)(L, H, D, B, plane_ptrs, int(num_blocks), p0, p1, int(first_token),
                              len(chunks), chunk_ptrs, ntok, bt.ctypes.data, bt.size)


def retrieve_fp8(L, H, D, B, planes, num_blocks, first_token, chunks, chunk_tokens, block_table,
                 p0=0, p1=None, lib=None) -> int:
    """Dequantising retrieval of one request: fp8 chunks (uint8 buffers) -> BF16 planes
    (uint16 arrays).  Returns 0, or -2 when a token has no valid block."""
    return _call_fp8("kvs_oracle_retrieve_fp8", L, H, D, B, planes, num_blocks, first_token,
                     chunks, chunk_tokens, block_table, p0, p1, lib)


def store_fp8(L, H, D, B, planes, num_blocks, first_token, chunks, chunk_tokens, block_table,
              p0=0, p1=None, lib=None) -> int:
    """Quantising store-back of one request: BF16 planes -> fp8 chunks (written in place)."""
    return _call_fp8("kvs_oracle_store_fp8", L, H, D, B, planes, num_blocks, first_token,
                     chunks, chunk_tokens, block_table, p0, p1, lib)
