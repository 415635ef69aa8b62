"""kvs_retrieve_noalloc, the retrieval entry point that allocates nothing.

Some callers cannot let a library allocate GPU memory: serving runtimes that
reserve nearly all free HBM for their own KV block pool at start-up and
sub-allocate it themselves (a cudaMalloc during serving could fail or break
their accounting), and latency-critical paths where cudaMalloc / cudaFree
would synchronise the device.  kvs_retrieve_noalloc keeps its scratch in a
static device array compiled into the library.

Its results are checked element by element against the CPU oracle (never
against another GPU path alone), on the random small geometries of the main
parity suite, capped grids, ragged last chunks, a shared-prefix batch of the
14B shape, and back-to-back calls without validation; two calls in a row must
also give exactly the bytes kvs_retrieve gives (the path only copies bytes, so
the tolerance is zero).  This file runs last, so a failure here comes after
every other test has run.
"""
import numpy as np
import pytest
import torch

import gpu_check as gc
from paper_2609_35065_gb300 import buffers, kvs, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    yield
    torch.cuda.synchronize()


def _noalloc(buf, flags=kvs.KVS_F_VALIDATE, stream=None):
    w = buf.workload
    return kvs.kvs_retrieve_noalloc(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, stream, flags)


def _mixed_shared_workload():
    # two requests with different residencies sharing their first two physical blocks
    g = synth.Geometry(4, 8, 128, 2, 16, 256)
    perm = np.random.default_rng(5).permutation(256).astype(np.int32)
    t0 = perm[:40]
    t1 = np.concatenate([t0[:2], perm[40:78]]).astype(np.int32)
    reqs = [synth.Request(640, 512, t0, "host"),
            synth.Request(608, 600, t1, "device", shared_prefix_tokens=32)]
    return synth.Workload("mixed_shared", g, 256, reqs, dist="normal", seed=11)


def _both_paths(w):
    buf = buffers.allocate(w)
    other = buf.planes.clone()
    g = w.geom
    ptrs_b = [int(other[p].data_ptr()) for p in range(other.shape[0])]
    kvs.kvs_retrieve(g, buf.plane_ptrs, w.num_blocks, buf.requests, None, kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    used_before = torch.cuda.memory_allocated()
    kvs.kvs_retrieve_noalloc(g, ptrs_b, w.num_blocks, buf.requests, None, kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    free_after = torch.cuda.mem_get_info()[0]
    assert torch.cuda.memory_allocated() == used_before
    return buf, other, free_before, free_after


def test_noalloc_matches_kvs_retrieve_and_the_oracle_on_two_calls_in_a_row():
    for k, w in enumerate([synth.tiny(), _mixed_shared_workload()]):
        buf, got, free_before, free_after = _both_paths(w)
        assert torch.equal(buf.planes, got), f"call {k + 1}: kvs_retrieve_noalloc differs from kvs_retrieve"
        assert not torch.all(got == got.view(-1)[0]), "nothing was written"
        buf.planes = got                       # the no-alloc result, element by element against the oracle
        gc.check_retrieve(buf)
        if k == 1:
            # the scratch array was set up on the first call; this call allocates nothing
            assert free_after >= free_before, (free_before, free_after)


@pytest.mark.parametrize("seed", range(40))
def test_noalloc_random_small_geometries_against_the_oracle(seed):
    w = gc.random_workload(seed)
    flags = [0, kvs.KVS_F_FORCE_HOSTLINK, kvs.KVS_F_FORCE_LDG, kvs.KVS_F_MAX_CTAS(1 + seed % 7)][seed % 4]
    buf = buffers.allocate(w)
    if seed % 2:
        _noalloc(buf, flags | kvs.KVS_F_VALIDATE)
    else:                                      # the unvalidated call: one synchronisation afterwards
        s = torch.cuda.Stream()
        _noalloc(buf, flags, s)
        s.synchronize()
    gc.check_retrieve(buf)


@pytest.mark.parametrize("residency", ["host", "device"])
@pytest.mark.parametrize("cap", [0, 7], ids=["default_grid", "max_ctas_7"])
def test_noalloc_capped_grids_and_ragged_last_chunks(residency, cap):
    """H8 D256: a block's run is 64 KiB (two pieces).  The 700-token request ends in a
    188-token chunk whose last block holds 12 tokens: full pieces, partial pieces and a
    partial block, on the link kernel (host chunks) or the vector kernel (device)."""
    w = synth.custom(2, 8, 256, 16, 256, 300, [1024, 700, 512], [1024, 700, 512], seed=5, dist="normal",
                     residency=residency)
    buf = buffers.allocate(w)
    _noalloc(buf, kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(cap))
    gc.check_retrieve(buf)


def test_noalloc_qwen14b_shaped_shared_prefix():
    """14B geometry (48 layers, 192 KiB per token), two requests of 12,288 matched tokens
    whose first 76 blocks are one shared physical run: written once, compared under
    KVS_F_VALIDATE, every element of all 96 planes against the oracle."""
    w = synth.qwen14b(requests=2, num_blocks=2048)
    assert w.notes["shared_blocks"] == 76
    buf = buffers.allocate(w, plane_init="random")
    _noalloc(buf)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.free(buf)


def test_noalloc_shared_blocks_with_differing_bytes_are_reported():
    buf = gc.shared_workload(differ=True)
    with pytest.raises(kvs.KvsError) as ei:
        _noalloc(buf)
    assert ei.value.code == kvs.KVS_ERR_ALIAS
    buf = gc.shared_workload(differ=False)
    _noalloc(buf)
    gc.check_retrieve(buf)


def test_noalloc_refuses_chunks_whose_memory_is_not_their_residency():
    """A pageable host buffer named as a pinned chunk, a pinned buffer named as a device
    chunk and a device buffer named as a pinned chunk are refused on the host before any
    work is enqueued: the planes keep their sentinel."""
    w = synth.tiny()
    buf = buffers.allocate(w)
    per_tok = 2 * w.geom.layers * w.geom.row_elems
    n = w.geom.chunk_tokens
    pageable = np.zeros(n * per_tok, dtype=np.int16)
    pinned = torch.zeros(n * per_tok, dtype=torch.int16, pin_memory=True)
    device = torch.zeros(n * per_tok, dtype=torch.int16, device="cuda")
    table = w.requests[0].block_table
    for base, res in [(pageable, kvs.KVS_SRC_HOST_PINNED), (pinned, kvs.KVS_SRC_DEVICE),
                      (device, kvs.KVS_SRC_HOST_PINNED)]:
        req = kvs.RequestArg(table, [kvs.ChunkArg(base, n, res)])
        with pytest.raises(kvs.KvsError) as ei:
            kvs.kvs_retrieve_noalloc(w.geom, buf.plane_ptrs, w.num_blocks, [req], None, 0)
        assert ei.value.code == kvs.KVS_ERR_INVALID_ARG, str(ei.value)
    torch.cuda.synchronize()
    assert torch.all(buf.planes == buf.planes.view(-1)[0])


def test_noalloc_back_to_back_calls_without_validation():
    """Three unvalidated calls, queued on one stream behind a ~50 ms sleep kernel, with
    different block tables into separate plane sets: each call refills the host staging
    tables while the previous uploads are still queued.  One synchronisation, then each
    result against the oracle."""
    bufs = [buffers.allocate(synth.custom(3, 4, 64, 16, 256, 200, [900, 640], [768, 600], seed=20 + k,
                                          residency=["host", "device"][k % 2]))
            for k in range(3)]
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        torch.cuda._sleep(100_000_000)
    for b in bufs:
        _noalloc(b, 0, s)
    s.synchronize()
    for b in bufs:
        gc.check_retrieve(b)


def test_noalloc_refuses_calls_beyond_its_scratch():
    # 4096-token chunks of 1-token blocks: 16 KiB of block ids per chunk, 80 chunks > 1 MiB.
    # Every address is a live buffer of the extent the call declares (planes 2 x 5 MiB,
    # chunks 80 x 128 KiB); the refusal comes before any of them is used.
    g = (1, 1, 8, 2, 1, 4096)
    nb = 80 * 4096
    planes = torch.zeros((2, nb * 8), dtype=torch.int16, device="cuda")
    chunk_elems = 2 * 4096 * 8
    pool = torch.zeros(80 * chunk_elems, dtype=torch.int16, pin_memory=True)
    chunks = [kvs.ChunkArg(pool[j * chunk_elems:(j + 1) * chunk_elems], 4096) for j in range(80)]
    req = kvs.RequestArg(np.arange(nb, dtype=np.int32), chunks)
    ptrs = [int(planes[0].data_ptr()), int(planes[1].data_ptr())]
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_noalloc(g, ptrs, nb, [req], None, 0)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    assert "KVS_NOALLOC_SCRATCH_BYTES" in str(ei.value)
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_noalloc(g, ptrs, nb, [req], None, kvs.KVS_F_FORCE_HBMCOPY)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert int(planes.abs().sum()) == 0


def test_noalloc_after_shutdown_looks_the_scratch_up_again():
    buf = buffers.allocate(synth.tiny())
    _noalloc(buf)
    torch.cuda.synchronize()
    assert kvs.kvs_shutdown() == kvs.KVS_OK
    buf.planes.fill_(int(np.array([synth.SENTINEL_BF16], dtype=np.uint16).view(np.int16)[0]))
    torch.cuda.synchronize()
    _noalloc(buf)
    gc.check_retrieve(buf)
