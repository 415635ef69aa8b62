"""Python binding of the C ABI in ``include/kvs.h`` (ctypes; argument marshalling only).

Every function has the C name and forwards to ``libkvs.so``; every byte is moved
by the library's CUDA kernels or copy-engine transfers.  There is no fallback:
if the library cannot be loaded, :func:`lib` raises.

Buffers are passed as integer addresses or as objects with ``data_ptr()``
(torch tensors).  Streams are passed as integer ``cudaStream_t`` handles,
objects with ``cuda_stream`` (``torch.cuda.Stream``), or ``None`` / 0 for the
legacy default stream.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass, field
from typing import Sequence

import numpy as np

from . import build as _build

# ---- constants mirrored from kvs.h ----------------------------------------
KVS_OK = 0
KVS_ERR_INVALID_ARG = -1
KVS_ERR_BOUNDS = -2
KVS_ERR_ALIAS = -3
KVS_ERR_CUDA = -4
KVS_ERR_TIMEOUT = -5
KVS_ERR_NOMEM = -6
KVS_ERR_UNSUPPORTED = -7
ERROR_NAMES = {0: "KVS_OK", -1: "KVS_ERR_INVALID_ARG", -2: "KVS_ERR_BOUNDS", -3: "KVS_ERR_ALIAS",
               -4: "KVS_ERR_CUDA", -5: "KVS_ERR_TIMEOUT", -6: "KVS_ERR_NOMEM", -7: "KVS_ERR_UNSUPPORTED"}

KVS_SRC_HOST_PINNED = 1
KVS_SRC_DEVICE = 2

KVS_F_VALIDATE = 1 << 0
KVS_F_FORCE_HOSTLINK = 1 << 1
KVS_F_FORCE_HBMCOPY = 1 << 2
KVS_F_FORCE_LDG = 1 << 3
KVS_F_FORCE_TMA = 1 << 4
KVS_F_NO_DEDUP = 1 << 5
KVS_F_LAYER_LAUNCHES = 1 << 6
KVS_F_LAYER_SIGNAL = 1 << 7
KVS_F_FORCE_DMA = 1 << 8
KVS_F_PREFETCH_L2 = 1 << 9
KVS_F_FEW_SMS = 1 << 10
KVS_DIR_RETRIEVE = 0
KVS_DIR_STORE = 1


def KVS_F_MAX_CTAS(n: int) -> int:
    return (int(n) & 0xFFFF) << 16


KVS_VARIANT_HOSTLINK = 1
KVS_VARIANT_HBMCOPY = 2
KVS_VARIANT_DMA = 3
VARIANT_NAMES = {1: "hostlink", 2: "hbmcopy", 3: "dma"}
KVS_KERNEL_LDG = 1
KVS_KERNEL_TMA = 2

EXPORTED = ("kvs_retrieve", "kvs_store", "kvs_query_bw", "kvs_get_choice", "kvs_check_errors",
            "kvs_enqueue_error_read",
            "kvs_last_error", "kvs_shutdown", "kvs_version", "kvs_selftest_wait_timeout",
            "kvs_stat_launches", "kvs_retrieve_noalloc", "kvs_retrieve_layers", "kvs_store_layers",
            "kvs_retrieve_fp8", "kvs_store_fp8", "kvs_retrieve_fp8_layers", "kvs_store_fp8_layers", "kvs_tune",
            "kvs_tier_create", "kvs_tier_destroy", "kvs_tier_commit", "kvs_tier_staged",
            "kvs_tier_begin_retrieval", "kvs_tier_end_retrieval", "kvs_tier_cancel", "kvs_tier_ordinary",
            "kvs_tier_claim_state", "kvs_tier_object", "kvs_tier_stats_get", "kvs_tier_slot")
KVS_CLAIM_NONE, KVS_CLAIM_PLANNED, KVS_CLAIM_STAGING, KVS_CLAIM_STAGE_READY = 0, 1, 2, 3
KVS_CLAIM_TRANSFERRING, KVS_CLAIM_RELEASED, KVS_CLAIM_CANCELLED, KVS_CLAIM_ORDINARY = 4, 5, 6, 7
CLAIM_NAMES = {0: "None", 1: "Planned", 2: "Staging", 3: "StageReady", 4: "Transferring",
               5: "Released", 6: "Cancelled", 7: "Ordinary"}
KVS_NOALLOC_SCRATCH_BYTES = 1 << 20


def KVS_FP8_SCALE_BYTES(L: int, H: int) -> int:
    return (2 * L * H * 4 + 255) // 256 * 256


class KvsError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERROR_NAMES.get(code, code)}: {msg}")
        self.code = code


# ---- ctypes mirrors of the structs ----------------------------------------
class kvs_geometry(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("elem_bytes", ctypes.c_int32),
                ("block_size", ctypes.c_int32), ("chunk_tokens", ctypes.c_int32)]


class kvs_chunk(ctypes.Structure):
    _fields_ = [("base", ctypes.c_void_p), ("num_tokens", ctypes.c_int32), ("residency", ctypes.c_int32)]


class kvs_request(ctypes.Structure):
    _fields_ = [("first_token", ctypes.c_int64), ("num_tokens", ctypes.c_int64),
                ("chunks", ctypes.POINTER(kvs_chunk)), ("num_chunks", ctypes.c_int32),
                ("block_table_len", ctypes.c_int32), ("block_table", ctypes.POINTER(ctypes.c_int32))]


class kvs_paged_cache(ctypes.Structure):
    _fields_ = [("kv_planes", ctypes.POINTER(ctypes.c_void_p)), ("num_blocks", ctypes.c_int64)]


class kvs_bw_report(ctypes.Structure):
    _fields_ = [("hbm_copy_gbs", ctypes.c_double), ("h2d_copy_engine_gbs", ctypes.c_double),
                ("d2h_copy_engine_gbs", ctypes.c_double), ("zero_copy_read_gbs", ctypes.c_double),
                ("zero_copy_write_gbs", ctypes.c_double), ("retrieve_gbs", ctypes.c_double * 2),
                ("store_gbs", ctypes.c_double * 2), ("device_kernel_gbs", ctypes.c_double * 2),
                ("chosen_retrieve_host", ctypes.c_int32), ("chosen_store_host", ctypes.c_int32),
                ("chosen_kernel_device", ctypes.c_int32), ("num_sms", ctypes.c_int32),
                ("hostlink_ctas", ctypes.c_int32), ("store_ctas", ctypes.c_int32),
                ("probe_bytes", ctypes.c_int64), ("retrieve_dma_gbs", ctypes.c_double),
                ("store_dma_gbs", ctypes.c_double), ("few_sm_ctas", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("few_sm_gbs", ctypes.c_double)]

    def as_dict(self) -> dict:
        out = {}
        for name, _ in self._fields_:
            v = getattr(self, name)
            out[name] = list(v) if isinstance(v, ctypes.Array) else v
        return out


class kvs_tune_report(ctypes.Structure):
    _fields_ = [("gbs", ctypes.c_double * 3), ("host_bytes", ctypes.c_int64), ("chosen", ctypes.c_int32),
                ("direction", ctypes.c_int32), ("device_gbs", ctypes.c_double * 2), ("device_bytes", ctypes.c_int64),
                ("chosen_kernel_device", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class kvs_tier_config(ctypes.Structure):
    _fields_ = [("capacity_objects", ctypes.c_int64), ("budget_objects", ctypes.c_int64),
                ("object_bytes", ctypes.c_int64), ("arena", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class kvs_tier_object_info(ctypes.Structure):
    _fields_ = [("slot", ctypes.c_int64), ("pins", ctypes.c_int32), ("staging", ctypes.c_int32),
                ("resident", ctypes.c_int32), ("gpu_refs", ctypes.c_int32), ("lru", ctypes.c_uint64)]


class kvs_tier_stats(ctypes.Structure):
    _fields_ = [("resident", ctypes.c_int64), ("staging", ctypes.c_int64), ("protected_objects", ctypes.c_int64),
                ("free_slots", ctypes.c_int64), ("evictions", ctypes.c_int64), ("staged_reads", ctypes.c_int64),
                ("completed", ctypes.c_int64), ("protected_object_seconds", ctypes.c_double)]


# ---- library loading ------------------------------------------------------
_lock = threading.Lock()
_lib = None


def lib_path() -> str:
    return os.environ.get("KVS_LIBRARY", _build.LIB)


def lib():
    """Load ``libkvs.so`` (building it first if sources are newer).  Raises if impossible."""
    global _lib
    with _lock:
        if _lib is None:
            path = lib_path()
            if "KVS_LIBRARY" not in os.environ and _build.stale():
                _build.build_library()
            if not os.path.exists(path):
                raise ImportError(f"libkvs.so not found at {path}: build it with "
                                  "`python -m paper_2609_35065_gb300.build`")
            L = ctypes.CDLL(path)
            P = ctypes.c_void_p
            for name in ("kvs_retrieve", "kvs_store", "kvs_retrieve_noalloc", "kvs_retrieve_fp8", "kvs_store_fp8"):
                fn = getattr(L, name)
                fn.argtypes = [ctypes.POINTER(kvs_geometry), ctypes.POINTER(kvs_paged_cache),
                               ctypes.POINTER(kvs_request), ctypes.c_int32, P, ctypes.c_uint32]
                fn.restype = ctypes.c_int
            EVP = ctypes.POINTER(ctypes.c_void_p)
            L.kvs_retrieve_layers.argtypes = [ctypes.POINTER(kvs_geometry), ctypes.POINTER(kvs_paged_cache),
                                              ctypes.POINTER(kvs_request), ctypes.c_int32, ctypes.c_int32,
                                              EVP, P, ctypes.c_uint32]
            L.kvs_retrieve_layers.restype = ctypes.c_int
            L.kvs_store_layers.argtypes = [ctypes.POINTER(kvs_geometry), ctypes.POINTER(kvs_paged_cache),
                                           ctypes.POINTER(kvs_request), ctypes.c_int32, ctypes.c_int32,
                                           EVP, EVP, P, ctypes.c_uint32]
            L.kvs_store_layers.restype = ctypes.c_int
            L.kvs_retrieve_fp8_layers.argtypes = L.kvs_retrieve_layers.argtypes
            L.kvs_retrieve_fp8_layers.restype = ctypes.c_int
            L.kvs_store_fp8_layers.argtypes = L.kvs_store_layers.argtypes
            L.kvs_store_fp8_layers.restype = ctypes.c_int
            U64P, I64P, I32P = (ctypes.POINTER(ctypes.c_uint64), ctypes.POINTER(ctypes.c_int64),
                                ctypes.POINTER(ctypes.c_int32))
            tier_sigs = {
                "kvs_tier_create": [ctypes.POINTER(kvs_tier_config), ctypes.POINTER(P)],
                "kvs_tier_destroy": [P],
                "kvs_tier_commit": [P, ctypes.c_uint64, U64P, ctypes.c_int32, ctypes.c_double, U64P, I32P],
                "kvs_tier_ordinary": [P, ctypes.c_uint64, U64P, ctypes.c_int32, ctypes.c_double, U64P, I32P],
                "kvs_tier_staged": [P, ctypes.c_uint64, ctypes.c_double],
                "kvs_tier_begin_retrieval": [P, ctypes.c_uint64, ctypes.c_double, I64P],
                "kvs_tier_end_retrieval": [P, ctypes.c_uint64, ctypes.c_double],
                "kvs_tier_cancel": [P, ctypes.c_uint64, ctypes.c_double],
                "kvs_tier_claim_state": [P, ctypes.c_uint64],
                "kvs_tier_object": [P, ctypes.c_uint64, ctypes.POINTER(kvs_tier_object_info)],
                "kvs_tier_stats_get": [P, ctypes.c_double, ctypes.POINTER(kvs_tier_stats)],
            }
            for name, sig in tier_sigs.items():
                fn = getattr(L, name)
                fn.argtypes = sig
                fn.restype = ctypes.c_int
            L.kvs_tier_slot.argtypes = [P, ctypes.c_int64]
            L.kvs_tier_slot.restype = ctypes.c_void_p
            L.kvs_tune.argtypes = [ctypes.POINTER(kvs_geometry), ctypes.POINTER(kvs_paged_cache),
                                   ctypes.POINTER(kvs_request), ctypes.c_int32, P, ctypes.c_uint32,
                                   ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(kvs_tune_report)]
            L.kvs_tune.restype = ctypes.c_int
            L.kvs_query_bw.argtypes = [ctypes.POINTER(kvs_bw_report), P, ctypes.c_int64]
            L.kvs_query_bw.restype = ctypes.c_int
            L.kvs_get_choice.argtypes = [ctypes.POINTER(kvs_bw_report)]
            L.kvs_get_choice.restype = ctypes.c_int
            L.kvs_check_errors.argtypes = [P]
            L.kvs_check_errors.restype = ctypes.c_int
            L.kvs_enqueue_error_read.argtypes = [P, P]
            L.kvs_enqueue_error_read.restype = ctypes.c_int
            L.kvs_last_error.argtypes = []
            L.kvs_last_error.restype = ctypes.c_char_p
            L.kvs_shutdown.argtypes = []
            L.kvs_shutdown.restype = ctypes.c_int
            L.kvs_version.argtypes = []
            L.kvs_version.restype = ctypes.c_int
            L.kvs_stat_launches.argtypes = []
            L.kvs_stat_launches.restype = ctypes.c_int64
            L.kvs_selftest_wait_timeout.argtypes = [P, ctypes.c_int64]
            L.kvs_selftest_wait_timeout.restype = ctypes.c_int
            _lib = L
    return _lib


# ---- marshalling helpers --------------------------------------------------
def _addr(x) -> int:
    if type(x) is int:
        return x
    ptr = getattr(x, "data_ptr", None)
    if ptr is not None:
        return int(ptr())
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        return int(x.ctypes.data)
    raise TypeError(f"cannot take the address of {type(x)!r}")


def _stream(s) -> int:
    if s is None:
        return 0
    if isinstance(s, int):
        return s
    if hasattr(s, "cuda_stream"):
        return int(s.cuda_stream)
    raise TypeError(f"not a stream: {type(s)!r}")


@dataclass
class ChunkArg:
    base: object                # address or tensor, [L][2][num_tokens][H][D]
    num_tokens: int
    residency: int = KVS_SRC_HOST_PINNED


@dataclass
class RequestArg:
    block_table: np.ndarray     # int32 physical block ids (host)
    chunks: Sequence[ChunkArg] = field(default_factory=list)
    first_token: int = 0
    num_tokens: int | None = None   # default: sum of chunk token counts


def _geometry(g) -> kvs_geometry:
    if isinstance(g, kvs_geometry):
        return g
    if hasattr(g, "layers"):
        return kvs_geometry(g.layers, g.kv_heads, g.head_dim, g.elem_bytes, g.block_size, g.chunk_tokens)
    return kvs_geometry(*g)


# numpy mirrors of kvs_chunk / kvs_request: one vectorised fill per call
_CHUNK_DT = np.dtype([("base", "<u8"), ("num_tokens", "<i4"), ("residency", "<i4")])
_REQ_DT = np.dtype([("first_token", "<i8"), ("num_tokens", "<i8"), ("chunks", "<u8"),
                    ("num_chunks", "<i4"), ("block_table_len", "<i4"), ("block_table", "<u8")])
assert _CHUNK_DT.itemsize == ctypes.sizeof(kvs_chunk) and _REQ_DT.itemsize == ctypes.sizeof(kvs_request)


class _Marshalled:
    """The C call's argument arrays (kept alive for the duration of one call)."""

    def __init__(self, planes, num_blocks, requests):
        if planes and all(type(p) is int for p in planes):
            self.planes = np.array(planes, dtype=np.uint64)
        else:
            self.planes = np.array([_addr(p) for p in planes] or [0], dtype=np.uint64)
        self.cache = kvs_paged_cache(ctypes.cast(int(self.planes.ctypes.data), ctypes.POINTER(ctypes.c_void_p)),
                                     int(num_blocks))
        counts = [len(r.chunks) for r in requests]
        chunks = np.zeros(max(1, sum(counts)), dtype=_CHUNK_DT)
        flat = [c for r in requests for c in r.chunks]
        if flat:
            chunks["base"] = [_addr(c.base) for c in flat]
            chunks["num_tokens"] = [c.num_tokens for c in flat]
            chunks["residency"] = [c.residency for c in flat]
        self.chunks = chunks
        self.tables = [np.ascontiguousarray(r.block_table, dtype=np.int32) for r in requests]
        reqs = np.zeros(max(1, len(requests)), dtype=_REQ_DT)
        if requests:
            base, step, at, starts = chunks.ctypes.data, _CHUNK_DT.itemsize, 0, []
            for n in counts:                          # address of each request's first chunk
                starts.append(base + at * step)
                at += n
            reqs["first_token"] = [r.first_token for r in requests]
            reqs["num_tokens"] = [sum(c.num_tokens for c in r.chunks) if r.num_tokens is None else r.num_tokens
                                  for r in requests]
            reqs["chunks"] = starts
            reqs["num_chunks"] = counts
            reqs["block_table_len"] = [t.size for t in self.tables]
            reqs["block_table"] = [t.ctypes.data for t in self.tables]
        self.reqs_np = reqs
        self.reqs = ctypes.cast(int(reqs.ctypes.data), ctypes.POINTER(kvs_request))
        self.n = len(requests)


def _check(rc: int) -> int:
    if rc != KVS_OK:
        raise KvsError(rc, lib().kvs_last_error().decode(errors="replace"))
    return rc


# ---- the C ABI, same names ------------------------------------------------
def kvs_retrieve(geom, planes, num_blocks, requests, stream=None, flags: int = 0) -> int:
    """Enqueue retrieval of ``requests`` (list of :class:`RequestArg`) into the 2L
    ``planes`` on ``stream``.  Raises :class:`KvsError` on a non-zero status."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    return _check(lib().kvs_retrieve(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                     _stream(stream), ctypes.c_uint32(flags)))


def kvs_store(geom, planes, num_blocks, requests, stream=None, flags: int = 0) -> int:
    """Enqueue store-back of ``requests`` from the planes into their chunk buffers."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    return _check(lib().kvs_store(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                  _stream(stream), ctypes.c_uint32(flags)))


def _events(events, stream):
    """cudaEvent_t handles of ``events``.  torch creates an event's handle at its first
    record, so a fresh ``torch.cuda.Event`` is first recorded once on the current
    stream; the library's record, made later in host order, is the one that waits see."""
    if events is None:
        return None, None
    handles = []
    for e in events:
        if e is None:
            handles.append(0)
        elif hasattr(e, "cuda_event"):
            if not int(e.cuda_event):
                import torch
                e.record(torch.cuda.current_stream())
            handles.append(int(e.cuda_event))
        else:
            handles.append(int(e))
    arr = (ctypes.c_void_p * max(1, len(handles)))(*handles)
    return arr, ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))


def kvs_retrieve_layers(geom, planes, num_blocks, requests, layers_per_step, layer_events=None,
                        stream=None, flags: int = 0) -> int:
    """Layer-wise :func:`kvs_retrieve`: ``layer_events[k]`` (``torch.cuda.Event`` or raw
    ``cudaEvent_t``) is recorded on ``stream`` after layer group k is enqueued."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    keep, ev = _events(layer_events, stream)
    return _check(lib().kvs_retrieve_layers(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                            int(layers_per_step), ev, _stream(stream), ctypes.c_uint32(flags)))


def _wait_events(events):
    """cudaEvent_t handles of events to wait on; an event never recorded (no handle yet)
    has nothing to wait for and is passed as NULL."""
    if events is None:
        return None, None
    handles = [0 if e is None else int(e.cuda_event) if hasattr(e, "cuda_event") else int(e) for e in events]
    arr = (ctypes.c_void_p * max(1, len(handles)))(*handles)
    return arr, ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))


def kvs_store_layers(geom, planes, num_blocks, requests, layers_per_step, layer_events=None,
                     stream=None, flags: int = 0, ready_events=None) -> int:
    """Layer-wise :func:`kvs_store`: group k waits on ``ready_events[k]`` (recorded by the
    caller once those layers' KV is computed) and records ``layer_events[k]`` when copied."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    keep_r, rev = _wait_events(ready_events)
    keep, ev = _events(layer_events, stream)
    return _check(lib().kvs_store_layers(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                         int(layers_per_step), rev, ev, _stream(stream), ctypes.c_uint32(flags)))


def kvs_query_bw(stream=None, probe_bytes: int = 0) -> dict:
    rep = kvs_bw_report()
    _check(lib().kvs_query_bw(ctypes.byref(rep), _stream(stream), int(probe_bytes)))
    return rep.as_dict()


def kvs_tune(geom, planes, num_blocks, requests, stream=None, flags: int = 0,
             direction: int = KVS_DIR_RETRIEVE, reps: int = 3) -> dict:
    """Time this call under each host-chunk variant, adopt the fastest as the default for
    its direction, and return {"gbs": [hostlink, hbmcopy, dma], "chosen": ..., ...}."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    rep = kvs_tune_report()
    _check(lib().kvs_tune(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n, _stream(stream),
                          ctypes.c_uint32(flags), int(direction), int(reps), ctypes.byref(rep)))
    return {"gbs": list(rep.gbs), "host_bytes": rep.host_bytes, "chosen": rep.chosen, "direction": rep.direction,
            "device_gbs": list(rep.device_gbs), "device_bytes": rep.device_bytes,
            "chosen_kernel_device": rep.chosen_kernel_device}


def kvs_get_choice() -> dict:
    rep = kvs_bw_report()
    _check(lib().kvs_get_choice(ctypes.byref(rep)))
    return rep.as_dict()


def kvs_check_errors(stream=None) -> int:
    return _check(lib().kvs_check_errors(_stream(stream)))


def kvs_enqueue_error_read(stream, host_word) -> int:
    """Enqueue a copy of the device error word into ``host_word`` (a pinned int32 tensor
    or address) and its reset, without synchronising; see kvs_check_errors."""
    return _check(lib().kvs_enqueue_error_read(_stream(stream), ctypes.c_void_p(_addr(host_word))))


def kvs_last_error() -> str:
    return lib().kvs_last_error().decode(errors="replace")


def kvs_shutdown() -> int:
    return _check(lib().kvs_shutdown())


def kvs_version() -> int:
    return int(lib().kvs_version())


def kvs_selftest_wait_timeout(stream=None, limit_ns: int = 50_000_000) -> int:
    """Runs the bounded-wait self-test; returns the status code (KVS_ERR_TIMEOUT expected)."""
    return int(lib().kvs_selftest_wait_timeout(_stream(stream), int(limit_ns)))


def kvs_stat_launches() -> int:
    return int(lib().kvs_stat_launches())


def kvs_retrieve_noalloc(geom, planes, num_blocks, requests, stream=None, flags: int = 0) -> int:
    """Like :func:`kvs_retrieve`, for callers that cannot let the library allocate GPU
    memory: its scratch is a static device array of KVS_NOALLOC_SCRATCH_BYTES, so the
    call allocates nothing; calls that overlap on the GPU race on that array."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    return _check(lib().kvs_retrieve_noalloc(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                             _stream(stream), ctypes.c_uint32(flags)))


def kvs_retrieve_fp8(geom, planes, num_blocks, requests, stream=None, flags: int = 0) -> int:
    """Dequantising retrieval from fp8 chunks (E4M3 codes with per-head scales) into
    BF16 planes; chunk buffers are [scales][codes], see kvs.h."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    return _check(lib().kvs_retrieve_fp8(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                         _stream(stream), ctypes.c_uint32(flags)))


def kvs_store_fp8(geom, planes, num_blocks, requests, stream=None, flags: int = 0) -> int:
    """Quantising store-back from BF16 planes into fp8 chunks (scales and codes written)."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    return _check(lib().kvs_store_fp8(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                      _stream(stream), ctypes.c_uint32(flags)))


def kvs_retrieve_fp8_layers(geom, planes, num_blocks, requests, layers_per_step, layer_events=None,
                            stream=None, flags: int = 0) -> int:
    """Layer-wise :func:`kvs_retrieve_fp8`; ``layer_events[k]`` is recorded after group k."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    keep, ev = _events(layer_events, stream)
    return _check(lib().kvs_retrieve_fp8_layers(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                                int(layers_per_step), ev, _stream(stream), ctypes.c_uint32(flags)))


def kvs_store_fp8_layers(geom, planes, num_blocks, requests, layers_per_step, layer_events=None,
                         stream=None, flags: int = 0, ready_events=None) -> int:
    """Layer-wise :func:`kvs_store_fp8`: group k waits on ``ready_events[k]``."""
    g = _geometry(geom)
    m = _Marshalled(planes, num_blocks, requests)
    keep_r, rev = _wait_events(ready_events)
    keep, ev = _events(layer_events, stream)
    return _check(lib().kvs_store_fp8_layers(ctypes.byref(g), ctypes.byref(m.cache), m.reqs, m.n,
                                             int(layers_per_step), rev, ev, _stream(stream), ctypes.c_uint32(flags)))


# ---- fast tier ------------------------------------------------------------
def _u64(keys):
    a = np.ascontiguousarray(np.asarray(keys, dtype=np.uint64))
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64))


class Tier:
    """The fast tier's ledger (and optional pinned arena): thin wrapper over kvs_tier_*.
    Every method takes the caller's clock ``now`` in seconds."""

    def __init__(self, capacity_objects: int, budget_objects: int, object_bytes: int, arena: bool = False):
        cfg = kvs_tier_config(int(capacity_objects), int(budget_objects), int(object_bytes), int(bool(arena)), 0)
        h = ctypes.c_void_p()
        _check(lib().kvs_tier_create(ctypes.byref(cfg), ctypes.byref(h)))
        self.handle = h
        self.object_bytes = int(object_bytes)

    def close(self):
        if self.handle:
            lib().kvs_tier_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _staging_call(self, fn, claim, keys, now):
        ks, kp = _u64(keys)
        out = np.zeros(max(1, ks.size), dtype=np.uint64)
        n = ctypes.c_int32(0)
        _check(fn(self.handle, int(claim), kp, int(ks.size), float(now),
                  out.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64)), ctypes.byref(n)))
        return [int(x) for x in out[:n.value]]

    def commit(self, claim, keys, now):
        """kvs_tier_commit: returns the keys whose staging the caller must now perform."""
        return self._staging_call(lib().kvs_tier_commit, claim, keys, now)

    def ordinary(self, claim, keys, now):
        """kvs_tier_ordinary: returns the keys to fetch on demand."""
        return self._staging_call(lib().kvs_tier_ordinary, claim, keys, now)

    def staged(self, key, now):
        _check(lib().kvs_tier_staged(self.handle, int(key), float(now)))

    def begin_retrieval(self, claim, now, n_keys):
        slots = np.zeros(max(1, n_keys), dtype=np.int64)
        _check(lib().kvs_tier_begin_retrieval(self.handle, int(claim), float(now),
                                              slots.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))))
        return [int(x) for x in slots[:n_keys]]

    def end_retrieval(self, claim, now):
        _check(lib().kvs_tier_end_retrieval(self.handle, int(claim), float(now)))

    def cancel(self, claim, now):
        _check(lib().kvs_tier_cancel(self.handle, int(claim), float(now)))

    def state(self, claim) -> int:
        return int(lib().kvs_tier_claim_state(self.handle, int(claim)))

    def object(self, key):
        info = kvs_tier_object_info()
        rc = lib().kvs_tier_object(self.handle, int(key), ctypes.byref(info))
        if rc == KVS_ERR_BOUNDS:
            return None
        _check(rc)
        return {"slot": info.slot, "pins": info.pins, "staging": info.staging, "resident": info.resident,
                "gpu_refs": info.gpu_refs, "lru": info.lru}

    def stats(self, now) -> dict:
        st = kvs_tier_stats()
        _check(lib().kvs_tier_stats_get(self.handle, float(now), ctypes.byref(st)))
        return {name: getattr(st, name) for name, _ in st._fields_}

    def slot_address(self, slot) -> int:
        return int(lib().kvs_tier_slot(self.handle, int(slot)) or 0)
