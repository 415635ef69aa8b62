"""GPU path (through the C ABI) against the CPU oracle, element by element.

Small cases span several 32 KiB pieces, ragged last chunks, B = 1, rows that
are not a multiple of 16 bytes, 1/2/4/8-byte elements, non-zero first tokens,
both residencies and every variant flag.  Exact equality is required: the
path only copies bytes.
"""
import numpy as np
import pytest
import torch

import gpu_check as gc
from paper_2609_35065_gb300 import buffers, kvs, synth

pytestmark = pytest.mark.gpu

VARIANTS = {
    "default": 0,
    "hostlink": kvs.KVS_F_FORCE_HOSTLINK,
    "hbmcopy": kvs.KVS_F_FORCE_HBMCOPY,
    "dma": kvs.KVS_F_FORCE_DMA,
    "ldg": kvs.KVS_F_FORCE_LDG,
    "tma": kvs.KVS_F_FORCE_TMA,
    "hbmcopy_tma": kvs.KVS_F_FORCE_HBMCOPY | kvs.KVS_F_FORCE_TMA,
    "few_ctas": kvs.KVS_F_MAX_CTAS(3),
    "tma_few_ctas": kvs.KVS_F_FORCE_TMA | kvs.KVS_F_MAX_CTAS(3),      # the persistent TMA pipeline
}


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    yield
    torch.cuda.synchronize()


def _retrieve(buf, flags=0, stream=None):
    w = buf.workload
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, stream, flags | kvs.KVS_F_VALIDATE)


def _store(buf, flags=0, stream=None):
    w = buf.workload
    kvs.kvs_store(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, stream, flags | kvs.KVS_F_VALIDATE)


def test_wait_timeout_selftest_then_context_usable():
    assert kvs.kvs_selftest_wait_timeout(None, 20_000_000) == kvs.KVS_ERR_TIMEOUT
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    buf = buffers.allocate(synth.tiny(), store=True)
    _retrieve(buf)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)


def test_enqueue_error_read_does_not_synchronise():
    """The status copy is queued behind the stream's work: the call returns while a
    ~50 ms sleep kernel still runs ahead of it, and the word reads 0 once it has run."""
    s = torch.cuda.Stream()
    word = torch.full((1,), -7, dtype=torch.int32, pin_memory=True)
    buf = buffers.allocate(synth.tiny(), store=True)
    w = buf.workload
    with torch.cuda.stream(s):
        torch.cuda._sleep(100_000_000)
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, 0)
    assert kvs.kvs_enqueue_error_read(s, word) == kvs.KVS_OK
    assert int(word[0]) == -7
    s.synchronize()
    assert int(word[0]) == kvs.KVS_OK
    gc.check_retrieve(buf)


@pytest.mark.parametrize("variant", sorted(VARIANTS))
def test_tiny_retrieve_then_store_round_trip(variant):
    flags = VARIANTS[variant]
    buf = buffers.allocate(synth.tiny(), store=True)
    _retrieve(buf, flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    _store(buf, flags)
    torch.cuda.synchronize()
    gc.check_store(buf)
    for a, b in zip(buf.chunks[0], buf.store_chunks[0]):        # store(retrieve(x)) == x
        assert torch.equal(a, b)


@pytest.mark.parametrize("variant", ["default", "hbmcopy", "tma", "tma_few_ctas"])
def test_tiny_device_resident_source(variant):
    w = synth.tiny()
    w.requests[0].residency = "device"
    buf = buffers.allocate(w, store=True, store_residency="device")
    _retrieve(buf, VARIANTS[variant])
    _store(buf, VARIANTS[variant])
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)


@pytest.mark.parametrize("seed", range(40))
def test_random_small_geometries(seed):
    w = gc.random_workload(seed)
    g = w.geom
    flags_all = [0, kvs.KVS_F_FORCE_HOSTLINK, kvs.KVS_F_FORCE_HBMCOPY, kvs.KVS_F_FORCE_LDG,
                 kvs.KVS_F_MAX_CTAS(1 + seed % 7)]
    row = g.row_elems * g.elem_bytes
    if row % 16 == 0:
        flags_all += [kvs.KVS_F_FORCE_TMA, kvs.KVS_F_FORCE_TMA | kvs.KVS_F_MAX_CTAS(2 + seed % 5)]
    flags = flags_all[seed % len(flags_all)]
    buf = buffers.allocate(w, store=True, store_residency="host" if seed % 2 else "device")
    _retrieve(buf, flags)
    _store(buf, flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)


@pytest.mark.parametrize("kernel", ["ldg", "tma", "ldg_capped", "tma_capped"])
@pytest.mark.parametrize("geometry", [(2, 8, 256), (3, 4, 128)], ids=["64KiB_runs", "16KiB_runs"])
def test_per_piece_kernels_full_and_partial_pieces(kernel, geometry):
    """Uncapped HBM copies run one CTA per 32 KiB piece; a CTA cap selects the grid-stride
    LDG kernel or the persistent TMA pipeline.  With H8 D256 a block's run is 64 KiB (two
    pieces); with H4 D128 it is 16 KiB (one short piece).  The 700-token request ends in a
    188-token chunk whose last block holds 12 tokens, so full pieces, partial pieces and
    partial blocks all occur, in both directions."""
    L, H, D = geometry
    flags = kvs.KVS_F_FORCE_LDG if kernel.startswith("ldg") else kvs.KVS_F_FORCE_TMA
    if kernel.endswith("capped"):
        flags |= kvs.KVS_F_MAX_CTAS(7)
    w = synth.custom(L, H, D, 16, 256, 300, [1024, 700, 512], [1024, 700, 512], seed=5, dist="normal",
                     residency="device")
    buf = buffers.allocate(w)
    _retrieve(buf, flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    ws = synth.custom(L, H, D, 16, 256, 300, [1024, 700], [0, 0], seed=6, store_tokens=[1024, 700])
    sbuf = buffers.allocate(ws, store=True, store_residency="device", plane_init="random")
    _store(sbuf, flags)
    torch.cuda.synchronize()
    gc.check_store(sbuf)


def test_tma_rejects_unaligned_rows():
    w = synth.custom(1, 3, 5, 4, 8, 8, [16], [16])            # 30-byte rows
    w.requests[0].residency = "device"
    buf = buffers.allocate(w)
    with pytest.raises(kvs.KvsError) as ei:
        _retrieve(buf, kvs.KVS_F_FORCE_TMA)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    assert torch.all(buf.planes == buf.planes.view(-1)[0])     # nothing written


@pytest.mark.parametrize("flags", [0, kvs.KVS_F_NO_DEDUP, kvs.KVS_F_FORCE_HBMCOPY])
def test_shared_blocks_written_once_with_equal_content(flags):
    buf = gc.shared_workload(differ=False)
    _retrieve(buf, flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)


def test_shared_blocks_with_differing_bytes_are_reported():
    buf = gc.shared_workload(differ=True)
    with pytest.raises(kvs.KvsError) as ei:
        _retrieve(buf)
    assert ei.value.code == kvs.KVS_ERR_ALIAS
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK            # the word was cleared


def test_block_named_twice_in_one_request_is_alias():
    w = synth.custom(1, 1, 8, 2, 4, 8, [8], [8])
    w.requests[0].block_table[1] = w.requests[0].block_table[0]
    buf = buffers.allocate(w)
    with pytest.raises(kvs.KvsError) as ei:
        _retrieve(buf)
    assert ei.value.code == kvs.KVS_ERR_ALIAS


def test_out_of_range_block_is_rejected_before_any_write():
    w = synth.custom(2, 2, 8, 4, 8, 8, [16], [16])
    w.requests[0].block_table[3] = 8
    buf = buffers.allocate(w)
    with pytest.raises(kvs.KvsError) as ei:
        _retrieve(buf)
    assert ei.value.code == kvs.KVS_ERR_BOUNDS
    torch.cuda.synchronize()
    assert torch.all(buf.planes == buf.planes.view(-1)[0])


def test_empty_calls_touch_nothing():
    w = synth.custom(2, 2, 8, 4, 8, 8, [16, 8], [0, 0])
    buf = buffers.allocate(w)
    _retrieve(buf)
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, [], None, kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    assert torch.all(buf.planes == buf.planes.view(-1)[0])


def test_streams_and_async_host_arrays():
    """The call returns before the copy runs; its host arrays may be dropped at once."""
    buf = buffers.allocate(synth.tiny())
    s = torch.cuda.Stream()
    w = buf.workload
    reqs = [kvs.RequestArg(r.block_table.copy(), list(r.chunks)) for r in buf.requests]
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, reqs, s, 0)
    for r in reqs:
        r.block_table[:] = -7                                   # reuse the host arrays
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve(buf)


def test_query_bw_reports_and_chooses():
    rep = kvs.kvs_query_bw(None, 256 << 20)
    for k in ("hbm_copy_gbs", "h2d_copy_engine_gbs", "d2h_copy_engine_gbs",
              "zero_copy_read_gbs", "zero_copy_write_gbs"):
        assert rep[k] > 1.0, (k, rep)
    assert rep["chosen_retrieve_host"] in (kvs.KVS_VARIANT_HOSTLINK, kvs.KVS_VARIANT_HBMCOPY)
    assert rep["chosen_kernel_device"] in (kvs.KVS_KERNEL_LDG, kvs.KVS_KERNEL_TMA)
    assert rep["num_sms"] > 0
    got = kvs.kvs_get_choice()
    assert got["chosen_retrieve_host"] == rep["chosen_retrieve_host"]
    # the chosen defaults still give exact results
    buf = buffers.allocate(synth.tiny(), store=True)
    _retrieve(buf)
    _store(buf)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)
