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
_SO = os.path.join(_HERE, "_build", "libkvs_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``kvs_oracle.c`` with gcc into ``oracle/_build`` (plain -O2, no tuning)."""
    os.makedirs(os.path.dirname(_SO), exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp], check=True)
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
