"""Host-chunk variants against the CPU oracle: the copy-engine DMA variant (2D copies
straight between chunks and planes), and kvs_tune, whose choice follows its own
measurement on the caller's call."""
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
    kvs.kvs_shutdown()                      # later tests start from the built-in defaults


def _sentinel(buf):
    buf.planes.fill_(int(np.array([synth.SENTINEL_BF16], dtype=np.uint16).view(np.int16)[0]))
    torch.cuda.synchronize()


@pytest.mark.parametrize("seed", range(12))
def test_dma_random_small_geometries(seed):
    """Retrieve and store with KVS_F_FORCE_DMA on the random geometries of the main suite
    (1/2/4/8-byte elements, B = 1..32, ragged last chunks, mixed residency: device chunks
    keep the SM kernel, host chunks go through 2D copies)."""
    w = gc.random_workload(seed)
    buf = buffers.allocate(w, store=True, store_residency="host")
    w_ = buf.workload
    kvs.kvs_retrieve(w_.geom, buf.plane_ptrs, w_.num_blocks, buf.requests, None,
                     kvs.KVS_F_FORCE_DMA | kvs.KVS_F_VALIDATE)
    kvs.kvs_store(w_.geom, buf.plane_ptrs, w_.num_blocks, buf.store_requests, None,
                  kvs.KVS_F_FORCE_DMA | kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)


def test_dma_shared_blocks_written_once():
    buf = gc.shared_workload(differ=False)
    w = buf.workload
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None,
                     kvs.KVS_F_FORCE_DMA | kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)


def test_dma_launches_no_kernel_for_host_chunks():
    buf = buffers.allocate(synth.tiny())
    w = buf.workload
    n0 = kvs.kvs_stat_launches()
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, kvs.KVS_F_FORCE_DMA)
    torch.cuda.synchronize()
    assert kvs.kvs_stat_launches() == n0
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    gc.check_retrieve(buf)


def test_dma_needs_equally_spaced_planes():
    """Planes from separate allocations: forcing DMA is refused before any copy; as a
    default it would fall back to the host-link kernel."""
    w = synth.tiny()
    buf = buffers.allocate(w)
    g = w.geom
    n = buf.planes.shape[1]
    planes = [torch.full((n,), int(buf.planes.view(-1)[0]), dtype=torch.int16, device="cuda")
              for _ in range(2 * g.layers)]
    ptrs = [int(p.data_ptr()) for p in planes][::-1]           # descending addresses
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve(g, ptrs, w.num_blocks, buf.requests, None, kvs.KVS_F_FORCE_DMA)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert all(torch.all(p == p[0]) for p in planes)


def test_dma_llama8b_batch():
    """The 4 GiB 8B batch from pinned host memory by 2048 2D copies, every element checked."""
    buf = buffers.allocate(synth.llama8b())
    w = buf.workload
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None,
                     kvs.KVS_F_FORCE_DMA | kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.free(buf)


@pytest.mark.parametrize("direction", [kvs.KVS_DIR_RETRIEVE, kvs.KVS_DIR_STORE], ids=["retrieve", "store"])
def test_tune_choice_follows_the_measurement(direction):
    """The host-link candidate is slowed on purpose (one CTA): the measured choice moves to
    a copy-engine variant, that variant then serves the next default call (the launch count
    tells which: DMA launches no kernel, HBMCOPY one scatter launch per ring batch), and the
    result equals the oracle's.  Tuned again without the cap, the choice is the measured best."""
    w = synth.llama8b(requests=2, num_blocks=1024)
    for r in w.requests:
        r.store_tokens, r.store_first = r.matched_tokens, 0
    buf = buffers.allocate(w, store=True)
    g = w.geom
    s = torch.cuda.Stream()
    reqs = buf.requests if direction == kvs.KVS_DIR_RETRIEVE else buf.store_requests
    if direction == kvs.KVS_DIR_STORE:        # the planes to store from: the retrieval's result
        kvs.kvs_retrieve(g, buf.plane_ptrs, w.num_blocks, buf.requests, s, kvs.KVS_F_VALIDATE)
    rep = kvs.kvs_tune(g, buf.plane_ptrs, w.num_blocks, reqs, s, kvs.KVS_F_MAX_CTAS(1), direction, reps=2)
    hostlink, hbmcopy, dma = rep["gbs"]
    assert rep["host_bytes"] == buf.payload_bytes
    assert min(hostlink, hbmcopy, dma) > 0, rep
    assert rep["chosen"] == [kvs.KVS_VARIANT_HOSTLINK, kvs.KVS_VARIANT_HBMCOPY,
                             kvs.KVS_VARIANT_DMA][int(np.argmax(rep["gbs"]))]
    assert rep["chosen"] != kvs.KVS_VARIANT_HOSTLINK, rep       # one CTA cannot keep up with the copy engine
    key = "chosen_retrieve_host" if direction == kvs.KVS_DIR_RETRIEVE else "chosen_store_host"
    assert kvs.kvs_get_choice()[key] == rep["chosen"]
    # the next default call runs the chosen variant, exactly
    if direction == kvs.KVS_DIR_RETRIEVE:
        _sentinel(buf)
    else:
        for mine in buf.store_chunks:
            for t in mine:
                t.fill_(0)
    n0 = kvs.kvs_stat_launches()
    fn = kvs.kvs_retrieve if direction == kvs.KVS_DIR_RETRIEVE else kvs.kvs_store
    fn(g, buf.plane_ptrs, w.num_blocks, reqs, s, 0)
    s.synchronize()
    launched = kvs.kvs_stat_launches() - n0
    assert launched == (0 if rep["chosen"] == kvs.KVS_VARIANT_DMA else 1) or \
        (rep["chosen"] == kvs.KVS_VARIANT_HBMCOPY and launched >= 1), (rep, launched)
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    if direction == kvs.KVS_DIR_RETRIEVE:
        gc.check_retrieve(buf)
    else:
        gc.check_store(buf)
    # uncapped, every candidate is measured again and the best one is taken
    rep2 = kvs.kvs_tune(g, buf.plane_ptrs, w.num_blocks, reqs, s, 0, direction, reps=2)
    assert rep2["chosen"] == [kvs.KVS_VARIANT_HOSTLINK, kvs.KVS_VARIANT_HBMCOPY,
                              kvs.KVS_VARIANT_DMA][int(np.argmax(rep2["gbs"]))]
    assert rep2["gbs"][0] > rep["gbs"][0]
    kvs.kvs_shutdown()
    gc.free(buf)


def test_tune_argument_checks():
    buf = buffers.allocate(synth.tiny())
    w = buf.workload
    for flags, direction, reps in [(kvs.KVS_F_FORCE_DMA, 0, 1), (0, 2, 1), (0, 0, 0), (kvs.KVS_F_FEW_SMS, 0, 1),
                                   (kvs.KVS_F_PREFETCH_L2, 0, 1)]:
        with pytest.raises(kvs.KvsError) as ei:
            kvs.kvs_tune(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, flags, direction, reps)
        assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
    # device-resident chunks only: the host-chunk choice is left alone
    w2 = synth.tiny()
    w2.requests[0].residency = "device"
    b2 = buffers.allocate(w2)
    before = kvs.kvs_get_choice()["chosen_retrieve_host"]
    rep = kvs.kvs_tune(w2.geom, b2.plane_ptrs, w2.num_blocks, b2.requests, None, 0, 0, 1)
    assert rep["host_bytes"] == 0 and rep["chosen"] == before and rep["gbs"] == [0, 0, 0]


@pytest.mark.parametrize("direction", [kvs.KVS_DIR_RETRIEVE, kvs.KVS_DIR_STORE], ids=["retrieve", "store"])
def test_tune_chooses_the_device_kernel_by_measurement(direction):
    """Mixed residency (the sweep's shape, scaled down): host chunks are tuned over the host
    variants, the device chunks alone over LDG and TMA; the faster kernel becomes the
    device default, and a default call afterwards equals the oracle."""
    w = synth.custom(4, 8, 128, 16, 256, 600, [2048, 2048, 1536, 1024], [1536, 1024, 1536, 768], seed=4,
                     dist="normal", residency=["host", "device", "device", "host"],
                     store_tokens=[256, 512, 0, 256])
    buf = buffers.allocate(w, store=True, store_residency="device")
    g = w.geom
    reqs = buf.requests if direction == kvs.KVS_DIR_RETRIEVE else buf.store_requests
    if direction == kvs.KVS_DIR_STORE:
        kvs.kvs_retrieve(g, buf.plane_ptrs, w.num_blocks, buf.requests, None, kvs.KVS_F_VALIDATE)
    rep = kvs.kvs_tune(g, buf.plane_ptrs, w.num_blocks, reqs, None, 0, direction, reps=2)
    assert rep["device_bytes"] > 0 and min(rep["device_gbs"]) > 0, rep
    want = kvs.KVS_KERNEL_TMA if rep["device_gbs"][1] > rep["device_gbs"][0] else kvs.KVS_KERNEL_LDG
    assert rep["chosen_kernel_device"] == want == kvs.kvs_get_choice()["chosen_kernel_device"]
    if direction == kvs.KVS_DIR_RETRIEVE:
        _sentinel(buf)
        kvs.kvs_retrieve(g, buf.plane_ptrs, w.num_blocks, reqs, None, kvs.KVS_F_VALIDATE)
        gc.check_retrieve(buf)
    else:
        for mine in buf.store_chunks:
            for t in mine:
                t.fill_(0)
        kvs.kvs_store(g, buf.plane_ptrs, w.num_blocks, reqs, None, kvs.KVS_F_VALIDATE)
        gc.check_store(buf)
    kvs.kvs_shutdown()


@pytest.mark.parametrize("cap", [0, 3, 12], ids=["default_grid", "3_ctas", "12_ctas"])
def test_prefetch_l2_retrieval(cap):
    """Host-link retrieval with L2 prefetches of each CTA's upcoming pieces: the 8B shape
    (2 requests, 512 MiB) and the ragged multi-piece shape, every element checked."""
    flags = kvs.KVS_F_PREFETCH_L2 | kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(cap)
    for w in (synth.llama8b(requests=2, num_blocks=1024),
              synth.custom(2, 8, 256, 16, 256, 300, [1024, 700, 512], [1024, 700, 512], seed=5, dist="normal")):
        buf = buffers.allocate(w)
        kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, flags)
        torch.cuda.synchronize()
        gc.check_retrieve(buf)
        gc.free(buf)


@pytest.mark.parametrize("seed", range(8))
def test_prefetch_l2_random_small_geometries(seed):
    """Random geometries: 16-byte rows take the prefetching kernel, the rest the vector
    kernel; stores ignore the flag."""
    w = gc.random_workload(seed)
    buf = buffers.allocate(w, store=True, store_residency="host")
    flags = kvs.KVS_F_PREFETCH_L2 | kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(seed % 3)
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, flags)
    kvs.kvs_store(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, None, flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)


@pytest.mark.parametrize("cap", [0, 1, 5, 20], ids=["default_grid", "1_cta", "5_ctas", "20_ctas"])
def test_few_sms_retrieval(cap):
    """KVS_F_FEW_SMS (one piece per thread in registers, three in shared memory): the 8B
    shape (2 requests, 512 MiB) and a ragged multi-piece shape, every element checked;
    one CTA cycles its four slots thousands of times."""
    flags = kvs.KVS_F_FEW_SMS | kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(cap)
    for w in (synth.llama8b(requests=2, num_blocks=1024),
              synth.custom(2, 8, 256, 16, 256, 300, [1024, 700, 512], [1024, 700, 512], seed=6, dist="normal")):
        buf = buffers.allocate(w)
        kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, flags)
        torch.cuda.synchronize()
        gc.check_retrieve(buf)
        gc.free(buf)


@pytest.mark.parametrize("seed", range(8))
def test_few_sms_random_small_geometries(seed):
    """Random geometries with mixed residency: 16-byte host rows take the staged kernel,
    the rest the vector kernel, device chunks their own kernels; stores ignore the flag."""
    w = gc.random_workload(seed)
    buf = buffers.allocate(w, store=True, store_residency="host")
    flags = kvs.KVS_F_FEW_SMS | kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(seed % 4)
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, flags)
    kvs.kvs_store(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, None, flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)


def test_few_sms_layerwise_groups_and_probe():
    """Layer-wise KVS_F_FEW_SMS retrieval (one staged launch per layer group) fires each
    group's event after exactly the oracle's planes of that group; kvs_query_bw then
    reports the staged kernel's cap and rate, and calls without a cap use it."""
    w = synth.custom(6, 8, 128, 16, 256, 200, [1024, 768], [1024, 768], seed=9)
    g = w.geom
    buf = buffers.allocate(w)
    events = [torch.cuda.Event() for _ in range(3)]
    copier, consumer = torch.cuda.Stream(), torch.cuda.Stream()
    kvs.kvs_retrieve_layers(g, buf.plane_ptrs, w.num_blocks, buf.requests, 2, events, copier, kvs.KVS_F_FEW_SMS)
    snaps = []
    for k, ev in enumerate(events):
        consumer.wait_event(ev)
        with torch.cuda.stream(consumer):
            snaps.append(buf.planes[4 * k:4 * k + 4].clone())
    torch.cuda.synchronize()
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    chunks_np = gc.host_chunks(buf)
    for k, snap in enumerate(snaps):
        for i in range(4):
            want = gc.expected_plane(buf, 4 * k + i, chunks_np)
            assert np.array_equal(snap[i].cpu().numpy().view(want.dtype), want), (k, i)
    rep = kvs.kvs_query_bw(None, 256 << 20)
    assert 10 <= rep["few_sm_ctas"] <= 40 and rep["few_sm_ctas"] % 2 == 0, rep["few_sm_ctas"]
    assert rep["few_sm_gbs"] > 0
    assert kvs.kvs_get_choice()["few_sm_ctas"] == rep["few_sm_ctas"]
    _sentinel(buf)
    kvs.kvs_retrieve(g, buf.plane_ptrs, w.num_blocks, buf.requests, None, kvs.KVS_F_FEW_SMS | kvs.KVS_F_VALIDATE)
    gc.check_retrieve(buf)
    kvs.kvs_shutdown()
