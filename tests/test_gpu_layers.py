"""Layer-wise retrieval / store-back through the C ABI, against the CPU oracle.

A consumer stream that waits on layer_events[k] must see layer group k
complete, whatever the later groups are doing; the final cache and stored
chunks must equal the oracle's on every element.
"""
import numpy as np
import pytest
import torch

import gpu_check as gc
import oracle
from paper_2609_35065_gb300 import buffers, kvs, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    yield
    torch.cuda.synchronize()


def _workload(residency="host", L=6):
    return synth.custom(L, 8, 128, 16, 256, 200, [1024, 768, 1280], [1024, 768, 1024], seed=8,
                        dist="normal", residency=residency)


@pytest.mark.parametrize("flags", [0, kvs.KVS_F_LAYER_SIGNAL, kvs.KVS_F_LAYER_SIGNAL | kvs.KVS_F_MAX_CTAS(4)],
                         ids=["launch_per_group", "signal", "signal_4ctas"])
@pytest.mark.parametrize("lps", [1, 2, 4, 6])
@pytest.mark.parametrize("residency", ["host", "device", "mixed"])
def test_layer_groups_are_ready_when_their_event_fires(lps, residency, flags):
    res = ["host", "device", "host"] if residency == "mixed" else residency
    w = _workload(res)
    g = w.geom
    buf = buffers.allocate(w)
    groups = -(-g.layers // lps)
    events = [torch.cuda.Event() for _ in range(groups)]
    copier, consumer = torch.cuda.Stream(), torch.cuda.Stream()
    kvs.kvs_retrieve_layers(g, buf.plane_ptrs, w.num_blocks, buf.requests, lps, events, copier, flags)
    snaps = []
    for k, ev in enumerate(events):
        consumer.wait_event(ev)
        p0, p1 = 2 * k * lps, 2 * min(g.layers, (k + 1) * lps)
        with torch.cuda.stream(consumer):
            snaps.append((p0, p1, buf.planes[p0:p1].clone()))
    torch.cuda.synchronize()
    chunks_np = gc.host_chunks(buf)
    for p0, p1, snap in snaps:
        for p in range(p0, p1):
            want = gc.expected_plane(buf, p, chunks_np)
            assert np.array_equal(snap[p - p0].cpu().numpy().view(np.uint16), want), (lps, p)
    gc.check_retrieve(buf, chunks_np=chunks_np)


def test_layerwise_equals_whole_call_with_validation_and_shared_blocks():
    g = synth.Geometry(4, 8, 128, 2, 16, 256)
    perm = np.random.default_rng(2).permutation(96).astype(np.int32)
    t0 = perm[:32]
    t1 = np.concatenate([t0[:4], perm[32:60]]).astype(np.int32)
    reqs = [synth.Request(512, 512, t0, "host"), synth.Request(512, 512, t1, "device", shared_prefix_tokens=64)]
    w = synth.Workload("layers_shared", g, 96, reqs, dist="normal", seed=4)
    a = buffers.allocate(w)
    b_planes = a.planes.clone()
    kvs.kvs_retrieve(g, a.plane_ptrs, w.num_blocks, a.requests, None, kvs.KVS_F_VALIDATE)
    ptrs = [int(b_planes[p].data_ptr()) for p in range(b_planes.shape[0])]
    kvs.kvs_retrieve_layers(g, ptrs, w.num_blocks, a.requests, 3, None, None, kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    assert torch.equal(a.planes, b_planes)
    gc.check_retrieve(a)


@pytest.mark.parametrize("lps", [1, 5])
def test_store_layers_matches_oracle(lps):
    """Host destinations with events: the signalling launch in the store direction."""
    w = synth.custom(5, 4, 64, 16, 256, 128, [1024, 700], [0, 0], seed=6, store_tokens=[768, 700])
    buf = buffers.allocate(w, store=True, plane_init="random")
    events = [torch.cuda.Event() for _ in range(-(-w.geom.layers // lps))]
    kvs.kvs_store_layers(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, lps, events, None,
                         kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    assert all(e.query() for e in events)
    gc.check_store(buf)


@pytest.mark.parametrize("dest", ["host", "device"])
@pytest.mark.parametrize("lps", [1, 2])
def test_store_layers_waits_for_each_groups_ready_event(lps, dest):
    """A producer stream rewrites layer group k's planes after a delay, then records
    ready[k]; the store must copy the rewritten bytes of every group (a store that did
    not wait would copy the planes' earlier contents)."""
    w = synth.custom(4, 8, 128, 16, 256, 128, [1024, 700], [0, 0], seed=11, store_tokens=[768, 700])
    g = w.geom
    buf = buffers.allocate(w, store=True, store_residency=dest, plane_init="random")
    groups = -(-g.layers // lps)
    gen = torch.Generator(device="cuda").manual_seed(3)
    fresh = torch.randint(-32768, 32767, tuple(buf.planes.shape), dtype=torch.int16, device="cuda", generator=gen)
    producer, copier = torch.cuda.Stream(), torch.cuda.Stream()
    ready = [torch.cuda.Event() for _ in range(groups)]
    torch.cuda.synchronize()
    with torch.cuda.stream(producer):
        for k in range(groups):
            torch.cuda._sleep(20_000_000)                 # ~10 ms: long after an unblocked copy
            p0, p1 = 2 * k * lps, 2 * min(g.layers, (k + 1) * lps)
            buf.planes[p0:p1].copy_(fresh[p0:p1])
            ready[k].record(producer)
    kvs.kvs_store_layers(g, buf.plane_ptrs, w.num_blocks, buf.store_requests, lps, None, copier,
                         kvs.KVS_F_VALIDATE, ready_events=ready)
    torch.cuda.synchronize()
    planes_np = [fresh[p].cpu().numpy().view(np.uint16) for p in range(2 * g.layers)]
    fill = synth.sentinel(2)
    for r, req in enumerate(buf.store_requests):
        want = [np.full(t.numel(), fill, dtype=np.uint16) for t in buf.store_chunks[r]]
        assert oracle.store(g.layers, g.kv_heads, g.head_dim, g.block_size, planes_np, w.num_blocks,
                            req.first_token, want, req.block_table) == 0
        for j, (t, e) in enumerate(zip(buf.store_chunks[r], want)):
            assert np.array_equal(t.cpu().numpy().view(np.uint16), e), (lps, r, j)


def test_empty_layerwise_call_still_records_events():
    w = _workload()
    buf = buffers.allocate(w)
    events = [torch.cuda.Event() for _ in range(3)]
    s = torch.cuda.Stream()
    kvs.kvs_retrieve_layers(w.geom, buf.plane_ptrs, w.num_blocks, [], 2, events, s, 0)
    s.synchronize()
    assert all(e.query() for e in events)
