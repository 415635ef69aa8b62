"""The C-ABI library without a GPU: it builds, loads, exports every function
declared in include/kvs.h, and rejects malformed calls before touching CUDA."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_35065_gb300 import kvs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "kvs.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(kvs_\w+)\s*\(", src, flags=re.M)))


def test_library_exports_every_declared_function():
    lib = kvs.lib()
    names = declared_functions()
    assert "kvs_retrieve" in names and "kvs_store" in names and "kvs_query_bw" in names
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(kvs.EXPORTED)
    assert kvs.kvs_version() == 10900


def test_struct_layouts_match_header():
    assert ctypes.sizeof(kvs.kvs_geometry) == 24
    assert ctypes.sizeof(kvs.kvs_chunk) == 16
    assert ctypes.sizeof(kvs.kvs_request) == 40
    assert ctypes.sizeof(kvs.kvs_paged_cache) == 16
    assert ctypes.sizeof(kvs.kvs_bw_report) == 5 * 8 + 6 * 8 + 6 * 4 + 8 + 2 * 8 + 2 * 4 + 8
    assert ctypes.sizeof(kvs.kvs_tune_report) == 3 * 8 + 8 + 2 * 4 + 2 * 8 + 8 + 2 * 4


class _Arena:
    """A live buffer for the addresses these tests pass, so that no call ever names
    memory that does not exist even if a validation check regressed: device memory
    (planes) or mapped pinned host memory (chunks) when a GPU is visible, plain host
    memory otherwise.  Every address handed out lies inside the buffer together with
    the whole extent the call declares for it."""

    def __init__(self, nbytes, kind):
        import torch
        if torch.cuda.is_available():
            self.t = (torch.zeros(nbytes, dtype=torch.uint8, device="cuda") if kind == "plane"
                      else torch.zeros(nbytes, dtype=torch.uint8, pin_memory=True))
            self.base = int(self.t.data_ptr())
        else:
            self.t = np.zeros(nbytes, dtype=np.uint8)
            self.base = int(self.t.ctypes.data)
        self.nbytes = nbytes

    def at(self, offset, extent):
        assert 0 <= offset and offset + extent <= self.nbytes, (offset, extent, self.nbytes)
        return self.base + offset


_arenas = {}


def arena(name, nbytes, kind):
    if name not in _arenas:
        _arenas[name] = _Arena(nbytes, kind)
    return _arenas[name]


G = (2, 2, 8, 2, 4, 8)          # rows of 32 B; a plane is 8 blocks x 4 rows = 1 KiB, a chunk of n tokens 4n rows
ROW = 32


def _planes(n=4):
    a = arena("planes", 64 << 10, "plane")
    return [a.at(4096 * p, 8 * 4 * ROW) for p in range(n)]


def _chunk(i, tokens):
    return arena("chunks", 64 << 10, "chunk").at(4096 * i, 4 * max(tokens, 0) * ROW)


def _req(tokens=(8, 8), table=(0, 1, 2, 3), first=0, res=kvs.KVS_SRC_HOST_PINNED, num_tokens=None):
    chunks = [kvs.ChunkArg(_chunk(i, n), n, res) for i, n in enumerate(tokens)]
    return kvs.RequestArg(np.array(table, np.int32), chunks, first, num_tokens)


def _code(fn=kvs.kvs_retrieve, geom=G, planes=None, nb=8, reqs=None, flags=0):
    """Status and message of one call (0 and "" when it succeeds)."""
    planes = _planes(2 * geom[0]) if planes is None else planes
    reqs = [_req()] if reqs is None else reqs
    try:
        fn(geom, planes, nb, reqs, None, flags)
    except kvs.KvsError as e:
        return e.code, str(e)
    return kvs.KVS_OK, ""


@pytest.mark.parametrize("fn", [kvs.kvs_retrieve, kvs.kvs_store])
@pytest.mark.parametrize("case,code", [
    (dict(geom=(0, 2, 8, 2, 4, 8)), kvs.KVS_ERR_INVALID_ARG),
    (dict(geom=(2, 2, 8, 3, 4, 8)), kvs.KVS_ERR_INVALID_ARG),          # 3-byte elements
    (dict(geom=(2, 2, 8, 2, 3, 8)), kvs.KVS_ERR_INVALID_ARG),          # C % B != 0
    (dict(nb=0), kvs.KVS_ERR_INVALID_ARG),
    (dict(planes="second_null"), kvs.KVS_ERR_INVALID_ARG),
    (dict(reqs=[_req(first=4)]), kvs.KVS_ERR_INVALID_ARG),             # not chunk-aligned
    (dict(reqs=[_req(tokens=(4, 8))]), kvs.KVS_ERR_INVALID_ARG),       # partial chunk not last
    (dict(reqs=[_req(tokens=(8, 9))]), kvs.KVS_ERR_INVALID_ARG),       # chunk larger than C
    (dict(reqs=[_req(num_tokens=12)]), kvs.KVS_ERR_INVALID_ARG),       # chunks hold 16
    (dict(reqs=[_req(res=7)]), kvs.KVS_ERR_INVALID_ARG),
    (dict(reqs=[_req(table=(0, 1, 2))]), kvs.KVS_ERR_BOUNDS),          # table too short
    (dict(reqs=[_req(table=(0, 1, 8, 3))]), kvs.KVS_ERR_BOUNDS),       # id >= num_blocks
    (dict(reqs=[_req(table=(0, -1, 2, 3))]), kvs.KVS_ERR_BOUNDS),
    (dict(flags=kvs.KVS_F_FORCE_HOSTLINK | kvs.KVS_F_FORCE_HBMCOPY), kvs.KVS_ERR_INVALID_ARG),
    (dict(flags=kvs.KVS_F_FORCE_LDG | kvs.KVS_F_FORCE_TMA), kvs.KVS_ERR_INVALID_ARG),
])
def test_malformed_calls_are_rejected(fn, case, code):
    if case.get("planes") == "second_null":
        p = _planes()
        case = dict(planes=[p[0], 0, p[2], p[3]])
    got, msg = _code(fn=fn, **case)
    assert got == code, msg
    assert kvs.kvs_last_error() == msg.split(": ", 1)[1]


@pytest.mark.parametrize("extra", [kvs.KVS_F_FORCE_HBMCOPY, kvs.KVS_F_FORCE_DMA, kvs.KVS_F_PREFETCH_L2],
                         ids=["hbmcopy", "dma", "prefetch_l2"])
def test_few_sms_retrieval_refuses_other_variants(extra):
    """KVS_F_FEW_SMS selects the host-link variant on its own kernel: combined with a
    copy-engine variant or the L2-prefetch kernel a retrieval is refused before any device
    work; a store ignores the flag (its argument checks still run first)."""
    got, msg = _code(fn=kvs.kvs_retrieve, flags=kvs.KVS_F_FEW_SMS | extra)
    assert got == kvs.KVS_ERR_INVALID_ARG, msg
    assert "KVS_F_FEW_SMS" in msg
    got, msg = _code(fn=kvs.kvs_store, reqs=[_req(table=(0, 1, 8, 3))], flags=kvs.KVS_F_FEW_SMS | extra)
    assert got == kvs.KVS_ERR_BOUNDS, msg


def test_few_sms_layerwise_refuses_the_signalling_launch():
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_layers(G, _planes(), 8, [_req()], 1, None, None, kvs.KVS_F_FEW_SMS | kvs.KVS_F_LAYER_SIGNAL)
    assert ei.value.code == kvs.KVS_ERR_INVALID_ARG


def test_null_base_pointer_is_rejected():
    r = _req()
    r.chunks[0].base = 0
    got, _ = _code(reqs=[r])
    assert got == kvs.KVS_ERR_INVALID_ARG


@pytest.mark.parametrize("fn,planes,reqs,alias", [
    # two planes on the same memory: retrieve writes both
    (kvs.kvs_retrieve, "0023", None, True),
    # the same for a store only reads them
    (kvs.kvs_store, "0023", None, False),
    # a source chunk inside a plane that the retrieve writes
    (kvs.kvs_retrieve, "0123", "chunk_in_plane", True),
    # store destinations overlapping each other (1 KiB chunks 512 B apart)
    (kvs.kvs_store, "0123", "chunks_overlap", True),
    # ... which a retrieve only reads
    (kvs.kvs_retrieve, "0123", "chunks_overlap", False),
], ids=["retrieve_planes", "store_planes", "retrieve_chunk_in_plane", "store_chunks", "retrieve_chunks"])
def test_validate_reports_overlapping_memory(fn, planes, reqs, alias):
    """With KVS_F_VALIDATE, memory a call writes may overlap neither itself nor what it
    reads (checked on the host before any device work)."""
    p = _planes()
    planes = [p[int(c)] for c in planes]
    r = _req()
    if reqs == "chunk_in_plane":
        # a 1 KiB chunk in the plane arena, starting inside plane 2 (1 KiB at 8 KiB)
        r.chunks[1].base = arena("planes", 64 << 10, "plane").at(2 * 4096 + 256, 1024)
        r.chunks[1].residency = kvs.KVS_SRC_DEVICE
    elif reqs == "chunks_overlap":
        r.chunks[1].base = arena("chunks", 64 << 10, "chunk").at(512, 1024)
    got, msg = _code(fn=fn, planes=planes, reqs=[r], flags=kvs.KVS_F_VALIDATE)
    if alias:
        assert got == kvs.KVS_ERR_ALIAS and "overlaps" in msg, msg
    else:
        # passes the check: succeeds with a GPU, fails later (no device) without one
        assert got != kvs.KVS_ERR_ALIAS, msg


def test_call_too_large_is_rejected():
    # 2^31 pieces or more: 32768 layers, 2-byte rows, B = 1, 128 chunks of 256 tokens.
    # Every plane is the same 64 KiB buffer (32768 blocks x 2 B) and every chunk the same
    # 32 MiB buffer (65536 planes x 256 tokens x 2 B): live memory of the declared extents.
    geom = (32768, 1, 1, 2, 1, 256)
    nb = 256 * 128
    plane = arena("too_large_plane", nb * 2, "plane").at(0, nb * 2)
    chunk_bytes = 2 * 32768 * 256 * 2
    chunk = arena("too_large_chunk", chunk_bytes, "chunk").at(0, chunk_bytes)
    req = kvs.RequestArg(np.arange(nb, dtype=np.int32), [kvs.ChunkArg(chunk, 256) for _ in range(128)])
    got, msg = _code(geom=geom, planes=[plane] * (2 * 32768), nb=nb, reqs=[req])
    assert got == kvs.KVS_ERR_INVALID_ARG and "too large" in msg


def test_empty_call_needs_no_device():
    assert kvs.kvs_retrieve(G, _planes(), 8, [], None, 0) == kvs.KVS_OK
    assert kvs.kvs_store(G, _planes(), 8, [_req(tokens=(), table=())], None, 0) == kvs.KVS_OK


@pytest.mark.parametrize("fn", [kvs.kvs_retrieve_layers, kvs.kvs_store_layers])
def test_layerwise_argument_checks(fn):
    with pytest.raises(kvs.KvsError) as ei:
        fn(G, _planes(), 8, [_req()], 0)
    assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
    with pytest.raises(kvs.KvsError) as ei:
        fn(G, _planes(), 8, [_req()], 1, None, None, kvs.KVS_F_FORCE_HBMCOPY)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    with pytest.raises(kvs.KvsError) as ei:
        fn(G, _planes(), 8, [_req()], 1, None, None, kvs.KVS_F_LAYER_LAUNCHES | kvs.KVS_F_LAYER_SIGNAL)
    assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
    if fn is kvs.kvs_store_layers:
        with pytest.raises(kvs.KvsError) as ei:
            fn(G, _planes(), 8, [_req()], 1, None, None, kvs.KVS_F_LAYER_SIGNAL, ready_events=[None, None])
        assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
    with pytest.raises(kvs.KvsError) as ei:
        fn(G, _planes(), 8, [_req(table=(0, 1, 9, 3))], 1)
    assert ei.value.code == kvs.KVS_ERR_BOUNDS
    assert fn(G, _planes(), 8, [], 1) == kvs.KVS_OK          # nothing to copy, no events given


def test_the_abi_from_plain_c(tmp_path):
    """tests/c_abi_smoke.c, compiled as C99 against include/kvs.h and linked with
    libkvs.so, runs its checks without a GPU."""
    import os
    import shutil
    import subprocess
    from paper_2609_35065_gb300 import build
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    kvs.lib()                                               # builds the library if needed
    here = os.path.dirname(os.path.abspath(__file__))
    exe = str(tmp_path / "c_abi_smoke")
    subprocess.run([gcc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic",
                    "-I", os.path.join(os.path.dirname(here), "include"),
                    os.path.join(here, "c_abi_smoke.c"), build.LIB, "-o", exe,
                    "-Wl,-rpath," + os.path.dirname(build.LIB)], check=True)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert out.returncode == 0, (out.returncode, out.stderr)
    assert out.stdout.strip() == "ok"



@pytest.mark.parametrize("flags", [kvs.KVS_F_FORCE_HOSTLINK, kvs.KVS_F_FEW_SMS, kvs.KVS_F_PREFETCH_L2,
                                   kvs.KVS_F_LAYER_SIGNAL], ids=["force", "few_sms", "prefetch_l2", "layer"])
def test_tune_refuses_kernel_choice_flags_before_device_work(flags):
    """kvs_tune picks the variant itself: flags that would choose a kernel for it are
    refused on the host, with no GPU (its candidates would not carry them)."""
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_tune(G, _planes(), 8, [_req()], None, flags, kvs.KVS_DIR_RETRIEVE, 1)
    assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
