"""Asynchrony of the C ABI on the GPU: many calls in flight on several streams,
calls from several host threads, retrieval beside a GEMM on another stream, and
stream order after a call whose two source classes ran on different streams.
Every result is compared with the CPU oracle element by element."""
import threading

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


def _small(seed, residency="host"):
    return synth.custom(4, 4, 64, 16, 256, 96, [600, 512, 300], [512, 512, 256], seed=seed,
                        residency=residency)


def test_more_calls_in_flight_than_descriptor_slots():
    """Twelve calls on three streams without host synchronisation; each stream
    retrieves into its own cache (descriptor slots are reused while calls are queued)."""
    streams = [torch.cuda.Stream() for _ in range(3)]
    bufs = [buffers.allocate(_small(10 + k, "host" if k % 2 else "device")) for k in range(3)]
    for rep in range(4):
        for s, b in zip(streams, bufs):
            w = b.workload
            kvs.kvs_retrieve(w.geom, b.plane_ptrs, w.num_blocks, b.requests, s, 0)
    torch.cuda.synchronize()
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    for b in bufs:
        gc.check_retrieve(b)


def test_calls_from_several_host_threads():
    bufs = [buffers.allocate(_small(20 + k)) for k in range(4)]
    errors = []

    def worker(b):
        try:
            s = torch.cuda.Stream()
            w = b.workload
            for _ in range(5):
                kvs.kvs_retrieve(w.geom, b.plane_ptrs, w.num_blocks, b.requests, s, 0)
            s.synchronize()
        except Exception as e:                              # reported below
            errors.append(e)

    threads = [threading.Thread(target=worker, args=(b,)) for b in bufs]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for b in bufs:
        gc.check_retrieve(b)


@pytest.mark.parametrize("flags", [0, kvs.KVS_F_FEW_SMS], ids=["default", "few_sms"])
def test_retrieval_beside_a_gemm_loop_is_exact(flags):
    buf = buffers.allocate(synth.llama8b(requests=2, num_blocks=1024))
    w = buf.workload
    side = torch.cuda.Stream(priority=-1)
    a = torch.randn(4096, 4096, dtype=torch.bfloat16, device="cuda")
    c = torch.empty_like(a)
    for _ in range(20):
        torch.matmul(a, a, out=c)                           # queued on the main stream
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, side, flags)
    for _ in range(20):
        torch.matmul(a, a, out=c)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)


def test_mixed_call_joins_the_callers_stream():
    """A consumer queued on the caller's stream right after a mixed-residency call
    sees every byte (the device part ran on a library stream and was joined)."""
    w = synth.custom(4, 8, 128, 16, 256, 160, [1024, 1024, 512], [1024, 1024, 512], seed=3,
                     residency=["device", "host", "device"])
    buf = buffers.allocate(w)
    s = torch.cuda.Stream()
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, 0)
    with torch.cuda.stream(s):
        snap = buf.planes.clone()                           # ordered after the call on s only
    s.synchronize()
    buf.planes = snap
    gc.check_retrieve(buf)


def test_store_then_retrieve_round_trip_on_one_stream():
    """store (cache -> host chunks) then retrieve of those chunks into a second cache,
    queued back to back: the second cache equals the oracle's retrieval of the stored
    chunks' expected contents."""
    w = synth.custom(3, 4, 32, 8, 64, 72, [320, 200], [0, 0], seed=5, store_tokens=[320, 200])
    src = buffers.allocate(w, store=True, plane_init="random")
    g = w.geom
    s = torch.cuda.Stream()
    kvs.kvs_store(g, src.plane_ptrs, w.num_blocks, src.store_requests, s, 0)
    dst = torch.full_like(src.planes, synth.SENTINEL_BF16)
    ptrs = [int(dst[p].data_ptr()) for p in range(dst.shape[0])]
    kvs.kvs_retrieve(g, ptrs, w.num_blocks, src.store_requests, s, 0)
    s.synchronize()
    gc.check_store(src)
    # every slot the store read now holds the same bytes in dst as in src
    B, R = g.block_size, g.row_elems
    for r, req in zip(src.store_requests, w.requests):
        for t in range(req.store_start, req.store_start + req.store_tokens):
            slot = int(req.block_table[t // B]) * B + t % B
            assert torch.equal(dst[:, slot * R:(slot + 1) * R], src.planes[:, slot * R:(slot + 1) * R])
