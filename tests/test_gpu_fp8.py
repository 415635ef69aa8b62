"""fp8 chunks (E4M3 codes of the OCP OFP8 specification, revision 1.0, with per-head
binary32 scales) through the C ABI against the CPU oracle, element by element.

Retrieval dequantises into BF16 planes; store-back quantises BF16 planes into fp8
chunks.  Both sides run the same round-to-nearest-even definitions, so the
comparison is exact: planes bit for bit, chunks byte for byte (scales and codes).
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


def _retrieve(buf, flags=kvs.KVS_F_VALIDATE, stream=None):
    w = buf.workload
    kvs.kvs_retrieve_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, stream, flags)


def _store(buf, flags=kvs.KVS_F_VALIDATE, stream=None):
    w = buf.workload
    kvs.kvs_store_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, stream, flags)


@pytest.mark.parametrize("residency", ["host", "device"])
def test_fp8_small_retrieve_and_store(residency):
    """L2 H4 D64, two 256-token chunks: dequantise, then quantise the same tokens back."""
    w = synth.custom(2, 4, 64, 16, 256, 128, [512], [512], residency=residency, store_tokens=[0])
    w.requests[0].store_tokens = 512
    w.requests[0].store_first = 0
    buf = buffers.allocate_fp8(w, store=True, store_residency=residency)
    _retrieve(buf)
    torch.cuda.synchronize()
    gc.check_retrieve_fp8(buf)
    _store(buf)
    torch.cuda.synchronize()
    gc.check_store_fp8(buf)


@pytest.mark.parametrize("seed", range(24))
def test_fp8_random_small_geometries(seed):
    w = gc.random_fp8_workload(seed)
    flags = [kvs.KVS_F_VALIDATE, 0, kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(1 + seed % 5)][seed % 3]
    buf = buffers.allocate_fp8(w, store=True, store_residency="host" if seed % 2 else "device")
    s = torch.cuda.Stream()
    _retrieve(buf, flags, s)
    s.synchronize()
    gc.check_retrieve_fp8(buf)
    _store(buf, flags, s)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_store_fp8(buf)


def _bf16(x):
    return np.array(x, dtype=np.float32).view(np.uint32) >> 16


@pytest.mark.parametrize("store_residency", ["host", "device"])
def test_fp8_special_values(store_residency):
    """Retrieval: NaN codes, the largest codes, subnormal codes and signed zeros under
    NaN, infinite, zero, subnormal and huge scales.  Store-back (per-head register kernel
    to pinned host, staged kernel to HBM): planes holding NaN, infinities, signed zeros,
    BF16 subnormals, values at exact midpoints between E4M3 codes (a head whose amax is
    448 has scale 1), and magnitudes at and around 2^-10."""
    w = synth.custom(2, 2, 32, 16, 32, 8, [64], [32], store_tokens=[32])
    buf = buffers.allocate_fp8(w, store=True, store_residency=store_residency)
    ch = buf.chunks[0][0]
    # one scale per (plane, head): 4 planes x 2 heads
    scales = np.array([np.nan, np.inf, 0.0, 1e-40, 3e38, 1.0, -2.0, 0.5], dtype=np.float32)
    sb = kvs.KVS_FP8_SCALE_BYTES(2, 2)
    ch[:8 * 4].copy_(torch.from_numpy(scales.view(np.uint8)))
    codes = np.arange(256, dtype=np.uint8)
    body = np.resize(codes, ch.numel() - sb)
    ch[sb:].copy_(torch.from_numpy(body))
    torch.cuda.synchronize()
    _retrieve(buf)
    torch.cuda.synchronize()
    gc.check_retrieve_fp8(buf)
    # store-back of planes with special BF16 values
    rng = np.random.default_rng(3)
    mids = np.array([1.0625, 1.1875, 0.0009765625, -0.0009765625, 0.0014648438, 2 ** -10 * 1.0078125,
                     13.0, 15.0, 17.0, 19.0, 240.0, 272.0, 464.0, 0.01367, 1e-40, -1e-40], dtype=np.float32)
    special = np.concatenate([_bf16(mids), [0x7FC0, 0xFFC0, 0x7F80, 0xFF80, 0x0000, 0x8000, 0x0001, 0x8001]])
    small = special[special != _bf16([464.0])[0]]                     # nothing above 448 in head 0
    for p in range(4):
        plane = buf.planes[p].view(-1)
        vals = rng.choice(special, size=plane.numel()).astype(np.uint16).reshape(-1, 2, 32)
        vals[:, 0, :] = rng.choice(small, size=vals[:, 0, :].shape)
        # head 0 of every plane has amax exactly 448 (scale 1): its midpoints are exact ties
        vals[:, 0, 0] = 0x43E0                                        # bf16 448.0
        plane.copy_(torch.from_numpy(vals.reshape(-1).view(np.int16)))
    torch.cuda.synchronize()
    _store(buf)
    torch.cuda.synchronize()
    gc.check_store_fp8(buf)


@pytest.mark.parametrize("store_residency", ["host", "device"])
def test_fp8_llama8b_host_batch_retrieve_and_store(store_residency):
    """The 8B batch (16 requests x 2048 matched tokens, 128 chunks of 256 tokens: 2 GiB of
    codes + scale blocks in pinned host memory) dequantised into the 20,000-block cache,
    then stored back into fresh fp8 chunks, pinned (the per-head register kernel) or in HBM
    (the staged kernel, 65,536 heads over one CTA per SM); every plane and chunk against
    the oracle."""
    w = synth.llama8b()
    for r in w.requests:
        r.store_tokens = r.matched_tokens
        r.store_first = 0
    buf = buffers.allocate_fp8(w, store=True, store_residency=store_residency)
    assert buf.payload_bytes == 128 * (2048 + (16 << 20))
    s = torch.cuda.Stream()
    kvs.kvs_retrieve_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve_fp8(buf)
    kvs.kvs_store_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_store_fp8(buf)


def test_fp8_refusals():
    w = synth.custom(1, 2, 32, 16, 32, 8, [64, 64], [32, 32])
    buf = buffers.allocate_fp8(w)
    g = w.geom
    # a physical block named by two requests
    reqs = [buf.requests[0], kvs.RequestArg(buf.requests[0].block_table, buf.requests[1].chunks)]
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_fp8(g, buf.plane_ptrs, w.num_blocks, reqs, None, 0)
    assert ei.value.code == kvs.KVS_ERR_ALIAS
    # head_dim not a multiple of 16 (the planes are large enough for the smaller rows)
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_fp8((1, 2, 24, 2, 16, 32), buf.plane_ptrs, w.num_blocks, buf.requests[:1], None, 0)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_fp8(g, buf.plane_ptrs, w.num_blocks, buf.requests, None, kvs.KVS_F_FORCE_HBMCOPY)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert torch.all(buf.planes == buf.planes.view(-1)[0])


@pytest.mark.parametrize("residency", ["host", "device"])
def test_fp8_store_two_pass_for_large_heads(residency):
    """chunk_tokens x head_dim above what one CTA holds in registers (256 x 256 = 65,536
    elements per head): the store takes the two-pass kernel (one CTA per chunk and plane);
    a ragged last chunk and a partial last block included."""
    w = synth.custom(2, 2, 256, 16, 256, 120, [700, 300], [0, 0], seed=9, residency=residency,
                     store_tokens=[700, 300])
    buf = buffers.allocate_fp8(w, store=True, store_residency=residency)
    rng = torch.Generator(device="cuda").manual_seed(9)
    for p in range(buf.planes.shape[0]):
        synth.fill_values(buf.planes[p], "normal", rng)
    torch.cuda.synchronize()
    _store(buf)
    torch.cuda.synchronize()
    gc.check_store_fp8(buf)


def test_fp8_qwen14b_shape_retrieve_and_suffix_store():
    """48 layers (192 KiB of BF16 per token), two requests of 12,288 matched tokens
    (48 chunks each, 2.25 GiB of fp8 chunks in pinned host memory) dequantised, then the
    computed 4096-token suffix of each stored back into fp8 chunks; every element of all
    96 planes and every byte of the stored chunks against the oracle."""
    w = synth.qwen14b(requests=2, num_blocks=2048, shared_frac=0.0)
    assert w.notes["shared_blocks"] == 0
    buf = buffers.allocate_fp8(w, store=True)
    s = torch.cuda.Stream()
    kvs.kvs_retrieve_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve_fp8(buf)
    # the suffix blocks hold computed KV: seeded normal values in every plane
    gen = torch.Generator(device="cuda").manual_seed(14)
    for p in range(buf.planes.shape[0]):
        synth.fill_values(buf.planes[p], "normal", gen)
    torch.cuda.synchronize()
    kvs.kvs_store_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_store_fp8(buf)


@pytest.mark.parametrize("lps", [1, 3])
@pytest.mark.parametrize("residency", ["host", "mixed"])
def test_fp8_layer_groups_are_ready_when_their_event_fires(lps, residency):
    """Layer-wise fp8 retrieval: a consumer stream that waits on layer_events[k] sees
    group k dequantised exactly as the oracle's, whatever later groups are doing."""
    res = ["host", "device", "host"] if residency == "mixed" else residency
    w = synth.custom(5, 8, 128, 16, 256, 200, [1024, 768, 1280], [1024, 768, 1024], seed=8, residency=res)
    g = w.geom
    buf = buffers.allocate_fp8(w)
    groups = -(-g.layers // lps)
    events = [torch.cuda.Event() for _ in range(groups)]
    copier, consumer = torch.cuda.Stream(), torch.cuda.Stream()
    kvs.kvs_retrieve_fp8_layers(g, buf.plane_ptrs, w.num_blocks, buf.requests, lps, events, copier, 0)
    snaps = []
    for k, ev in enumerate(events):
        consumer.wait_event(ev)
        p0, p1 = 2 * k * lps, 2 * min(g.layers, (k + 1) * lps)
        with torch.cuda.stream(consumer):
            snaps.append((p0, p1, buf.planes[p0:p1].clone()))
    torch.cuda.synchronize()
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    chunks_np = [[gc._np(t) for t in mine] for mine in buf.chunks]
    for p0, p1, snap in snaps:
        for p in range(p0, p1):
            want = gc.expected_plane_fp8(buf, p, chunks_np)
            assert np.array_equal(snap[p - p0].cpu().numpy().view(np.uint16), want), (lps, p)
    gc.check_retrieve_fp8(buf, chunks_np=chunks_np)


def test_fp8_layerwise_store_waits_for_ready_events():
    """Layer-wise fp8 store-back: a producer rewrites each layer group's planes after a
    delay and then records its ready event; the stored chunks equal the oracle's store of
    the rewritten planes."""
    w = synth.custom(4, 8, 128, 16, 256, 200, [1024, 768], [0, 0], seed=12, store_tokens=[1024, 768])
    g = w.geom
    buf = buffers.allocate_fp8(w, store=True)
    lps = 2
    groups = -(-g.layers // lps)
    ready = [torch.cuda.Event() for _ in range(groups)]
    done = [torch.cuda.Event() for _ in range(groups)]
    producer, copier = torch.cuda.Stream(), torch.cuda.Stream()
    gen = torch.Generator(device="cuda").manual_seed(12)
    with torch.cuda.stream(producer):
        for k in range(groups):
            torch.cuda._sleep(20_000_000)
            for p in range(2 * k * lps, 2 * min(g.layers, (k + 1) * lps)):
                synth.fill_values(buf.planes[p], "normal", gen)
            ready[k].record(producer)
    kvs.kvs_store_fp8_layers(g, buf.plane_ptrs, w.num_blocks, buf.store_requests, lps, done, copier, 0,
                             ready_events=ready)
    torch.cuda.synchronize()
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    gc.check_store_fp8(buf)


def test_fp8_layerwise_argument_checks():
    w = synth.custom(2, 2, 32, 16, 32, 8, [64], [32])
    buf = buffers.allocate_fp8(w)
    for fn in (kvs.kvs_retrieve_fp8_layers, kvs.kvs_store_fp8_layers):
        with pytest.raises(kvs.KvsError) as ei:
            fn(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, 0)
        assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
        with pytest.raises(kvs.KvsError) as ei:
            fn(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, 1, None, None, kvs.KVS_F_LAYER_SIGNAL)
        assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED


@pytest.mark.parametrize("D,B", [(48, 3), (80, 16), (176, 1)])
def test_fp8_head_dims_that_are_not_powers_of_two(D, B):
    """head_dim 48 / 80 / 176 (3, 5 and 11 vectors of 16 codes per head): the retrieval's
    per-vector head arithmetic and the two-pass store (D/8 does not divide the CTA), with
    B = 3 and B = 1 paged blocks and a ragged last chunk, both residencies."""
    C = 48 if B == 3 else 64
    w = synth.custom(2, 3, D, B, C, 400, [200, 150], [150, 100], seed=D, residency=["host", "device"],
                     store_tokens=[0, 0])
    for r in w.requests:
        r.store_tokens, r.store_first = r.matched_tokens, r.first_token
    buf = buffers.allocate_fp8(w, store=True)
    _retrieve(buf)
    torch.cuda.synchronize()
    gc.check_retrieve_fp8(buf)
    _store(buf)
    torch.cuda.synchronize()
    gc.check_store_fp8(buf)


@pytest.mark.parametrize("ctas", [1, 2, 7])
def test_fp8_staged_store_with_few_ctas(ctas):
    """HBM-destination store-back with 1, 2 and 7 CTAs: each CTA cycles its shared-memory
    stages many times (stage reuse, barrier phases wrapping), over full chunks, a ragged
    last chunk and a nonzero store start."""
    w = synth.custom(3, 4, 128, 16, 256, 300, [1500, 1100], [0, 0], seed=ctas, store_tokens=[1200, 1000],
                     firsts=[256, 0])
    buf = buffers.allocate_fp8(w, store=True, store_residency="device")
    gen = torch.Generator(device="cuda").manual_seed(ctas)
    for p in range(buf.planes.shape[0]):
        synth.fill_values(buf.planes[p], "normal", gen)
    torch.cuda.synchronize()
    _store(buf, kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(ctas))
    torch.cuda.synchronize()
    gc.check_store_fp8(buf)


@pytest.mark.parametrize("store_residency", ["host", "device"])
def test_fp8_store_nan_without_infinity(store_residency):
    """Heads holding NaNs of both signs (and no infinity) among normal values, heads of
    zeros and BF16 subnormals only, and heads holding one infinity: the amax ignores the
    NaNs and infinities, and every code and scale equals the oracle's."""
    w = synth.custom(2, 8, 128, 16, 256, 64, [512], [0], seed=5, store_tokens=[512])
    buf = buffers.allocate_fp8(w, store=True, store_residency=store_residency)
    rng = np.random.default_rng(5)
    for p in range(buf.planes.shape[0]):
        vals = _bf16(rng.standard_normal(buf.planes[p].numel()).astype(np.float32)).astype(np.uint16)
        vals = vals.reshape(-1, 8, 128)                       # [rows][head][d]
        for h, kind in enumerate(["nan", "nan", "zero_sub", "inf", "nan_inf", "plain", "nan", "zero"]):
            sel = vals[:, h, :].copy()
            if kind.startswith("nan"):                        # ~2% NaNs of both signs
                idx = rng.choice(sel.size, size=sel.size // 50, replace=False)
                sel.reshape(-1)[idx] = rng.choice(np.array([0x7FC0, 0xFFC0, 0x7FC1, 0xFFFF, 0x7F81, 0xFF81],
                                                           dtype=np.uint16), size=idx.size)
            if kind.endswith("inf"):                          # ~0.05% infinities of both signs
                idx = rng.choice(sel.size, size=sel.size // 2000, replace=False)
                sel.reshape(-1)[idx] = rng.choice(np.array([0x7F80, 0xFF80], dtype=np.uint16), size=idx.size)
            if kind == "zero_sub":
                sel[:] = rng.choice(np.array([0x0000, 0x8000, 0x0001, 0x8003, 0x007F], dtype=np.uint16), size=sel.shape)
            if kind == "zero":
                sel[:] = 0
            vals[:, h, :] = sel
        buf.planes[p].copy_(torch.from_numpy(vals.reshape(-1).view(np.int16)))
    torch.cuda.synchronize()
    _store(buf)
    torch.cuda.synchronize()
    gc.check_store_fp8(buf)


@pytest.mark.parametrize("cap", [0, 1, 6], ids=["default_grid", "1_cta", "6_ctas"])
def test_fp8_few_sms_retrieval(cap):
    """KVS_F_FEW_SMS with fp8 chunks (two pieces of codes in registers and five in shared
    memory, scales copied per vector): the 8B batch shape (2 requests) and a mixed, ragged
    shape with an odd head count, every element against the oracle; stores ignore the flag."""
    flags = kvs.KVS_F_FEW_SMS | kvs.KVS_F_VALIDATE | kvs.KVS_F_MAX_CTAS(cap)
    for w in (synth.llama8b(requests=2, num_blocks=1024),
              synth.custom(3, 5, 48, 16, 64, 300, [700, 520, 400], [640, 448, 320], seed=cap,
                           residency=["host", "device", "host"], firsts=[0, 64, 0], store_tokens=[0, 0, 0])):
        buf = buffers.allocate_fp8(w)
        _retrieve(buf, flags)
        torch.cuda.synchronize()
        gc.check_retrieve_fp8(buf)


def test_fp8_few_sms_layer_groups():
    """Layer-wise fp8 retrieval on the few-SM kernel: each group's event fires after exactly
    the oracle's planes of that group."""
    w = synth.custom(4, 8, 128, 16, 256, 200, [1024, 768], [1024, 768], seed=21)
    g = w.geom
    buf = buffers.allocate_fp8(w)
    events = [torch.cuda.Event() for _ in range(2)]
    copier, consumer = torch.cuda.Stream(), torch.cuda.Stream()
    kvs.kvs_retrieve_fp8_layers(g, buf.plane_ptrs, w.num_blocks, buf.requests, 2, events, copier, kvs.KVS_F_FEW_SMS)
    snaps = []
    for k, ev in enumerate(events):
        consumer.wait_event(ev)
        with torch.cuda.stream(consumer):
            snaps.append(buf.planes[4 * k:4 * k + 4].clone())
    torch.cuda.synchronize()
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
    chunks_np = [[gc._np(t) for t in mine] for mine in buf.chunks]
    for k, snap in enumerate(snaps):
        for i in range(4):
            want = gc.expected_plane_fp8(buf, 4 * k + i, chunks_np)
            assert np.array_equal(snap[i].cpu().numpy().view(np.uint16), want), (k, i)


def test_fp8_llama8b_batch_few_sms():
    """The full 8B batch (128 fp8 chunks, 2 GiB of codes in pinned host memory) retrieved
    with KVS_F_FEW_SMS on its default cap after kvs_query_bw, as the overlap benchmark runs
    it; every plane against the oracle."""
    s = torch.cuda.Stream()
    kvs.kvs_query_bw(s, 256 << 20)
    w = synth.llama8b()
    buf = buffers.allocate_fp8(w)
    kvs.kvs_retrieve_fp8(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, kvs.KVS_F_FEW_SMS)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve_fp8(buf)
    kvs.kvs_shutdown()
