"""Full-size workloads through the C ABI, compared with the CPU oracle on every
element of every plane (streamed one plane at a time through the oracle)."""
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
    torch.cuda.empty_cache()


def _run(buf, fn="retrieve", flags=0):
    w = buf.workload
    reqs = buf.requests if fn == "retrieve" else buf.store_requests
    getattr(kvs, f"kvs_{fn}")(w.geom, buf.plane_ptrs, w.num_blocks, reqs, None, flags | kvs.KVS_F_VALIDATE)


@pytest.mark.parametrize("flags", [0, kvs.KVS_F_FORCE_HOSTLINK, kvs.KVS_F_FORCE_HBMCOPY],
                         ids=["default", "hostlink", "hbmcopy"])
def test_llama8b_host_source(flags):
    buf = buffers.allocate(synth.llama8b())
    assert buf.payload_bytes == 4 << 30
    _run(buf, flags=flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.free(buf)


def test_llama8b_in_the_bench_launch_configuration():
    """The calls bench.py times: after kvs_query_bw has chosen the variants and the
    host-link grid, flags 0 on a side stream (no validation pass), the host-source
    batch and then the same chunks staged in HBM; every element checked."""
    s = torch.cuda.Stream()
    choice = kvs.kvs_query_bw(s, 1 << 30)
    buf = buffers.allocate(synth.llama8b())
    w = buf.workload
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve(buf)
    # the same batch from an HBM staging copy of the chunks, into sentinel planes
    dpool = buf.host_pool.to("cuda")
    per_tok = 2 * w.geom.layers * w.geom.row_elems
    dreqs, at = [], 0
    for r in buf.requests:
        cs = []
        for c in r.chunks:
            cs.append(kvs.ChunkArg(dpool[at:at + c.num_tokens * per_tok], c.num_tokens, kvs.KVS_SRC_DEVICE))
            at += c.num_tokens * per_tok
        dreqs.append(kvs.RequestArg(r.block_table, cs, r.first_token))
    buf.planes.fill_(np.array([synth.SENTINEL_BF16], dtype=np.uint16).view(np.int16)[0].item())
    s.wait_stream(torch.cuda.current_stream())          # the refill runs on torch's stream
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, dreqs, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve(buf)
    assert choice["chosen_kernel_device"] in (kvs.KVS_KERNEL_LDG, kvs.KVS_KERNEL_TMA)
    del dpool
    gc.free(buf)


@pytest.mark.parametrize("ratio,flags", [(25, 0), (50, 0), (75, 0), (50, kvs.KVS_F_FORCE_TMA),
                                         (50, kvs.KVS_F_FORCE_LDG)],
                         ids=["25", "50", "75", "50_tma", "50_ldg"])
def test_sweep_mixed_residency(ratio, flags):
    """Host class on the host-link kernel, HBM class (one CTA per piece, LDG or TMA)
    beside it on a second stream."""
    w = synth.sweep(ratio / 100)
    res = {r.residency for r in w.requests}
    assert res == {"host", "device"}
    buf = buffers.allocate(w)
    _run(buf, flags=flags)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.free(buf)


def test_qwen14b_shared_prefix_retrieve_and_suffix_store():
    w = synth.qwen14b()
    assert w.notes["shared_blocks"] == 76
    buf = buffers.allocate(w, store=True, store_residency="host", plane_init="random")
    _run(buf, "retrieve")
    _run(buf, "store")
    torch.cuda.synchronize()
    chunks_np = gc.host_chunks(buf)
    gc.check_retrieve(buf, chunks_np=chunks_np)
    gc.check_store(buf, chunks_np=chunks_np)
    gc.free(buf)


def test_qwen14b_store_to_hbm_destination_hbmcopy_path():
    w = synth.qwen14b()
    buf = buffers.allocate(w, store=True, store_residency="device", plane_init="random")
    _run(buf, "retrieve", kvs.KVS_F_FORCE_HBMCOPY)
    _run(buf, "store", kvs.KVS_F_FORCE_TMA)
    torch.cuda.synchronize()
    chunks_np = gc.host_chunks(buf)
    gc.check_retrieve(buf, chunks_np=chunks_np)
    gc.check_store(buf, chunks_np=chunks_np)
    gc.free(buf)


@pytest.mark.parametrize("frac,flags", [(0.25, 0), (0.5, 0), (0.25, kvs.KVS_F_FEW_SMS)],
                         ids=["25pct", "50pct", "25pct_few_sms"])
def test_llama70b_partial_buffer_refilled_between_passes(frac, flags):
    """Pinned fast-tier buffer holds 25% (4 passes of one request) or 50% (2 passes of two
    requests) of the batch, refilled in between; every pass is one call (with
    KVS_F_FEW_SMS: the staged kernel on its cap, as the overlap benchmark runs it)."""
    w = synth.llama70b(buffer_frac=frac)
    g = w.geom
    per_tok = 2 * g.layers * g.row_elems
    per_pass = int(round(len(w.requests) * frac))
    n = w.num_blocks * g.block_size * g.row_elems
    planes = torch.full((2 * g.layers, n), synth.SENTINEL_BF16, dtype=torch.int16, device="cuda")
    ptrs = [int(planes[p].data_ptr()) for p in range(2 * g.layers)]
    one_req = w.requests[0].matched_tokens * per_tok
    pinned = torch.empty(per_pass * one_req, dtype=torch.int16, pin_memory=True)
    assert pinned.numel() * len(w.requests) == int(frac * len(w.requests)) * w.matched_tokens * per_tok
    host_copies = []
    for k in range(0, len(w.requests), per_pass):
        tmp = torch.empty(per_pass * one_req, dtype=torch.int16, device="cuda")
        synth.fill_values(tmp, "normal", torch.Generator(device="cuda").manual_seed(100 + k))
        torch.cuda.synchronize()
        pinned.copy_(tmp)                                   # refill between passes (untimed)
        del tmp
        reqs = []
        for i, r in enumerate(w.requests[k:k + per_pass]):
            base = i * one_req
            chunks = [pinned[base + j * 256 * per_tok:base + (j + 1) * 256 * per_tok]
                      for j in range(r.matched_tokens // 256)]
            reqs.append(kvs.RequestArg(r.block_table, [kvs.ChunkArg(c, 256) for c in chunks]))
            host_copies.append([c.numpy().copy().view(np.uint16) for c in chunks])
        kvs.kvs_retrieve(g, ptrs, w.num_blocks, reqs, None, kvs.KVS_F_VALIDATE | flags)
        torch.cuda.synchronize()
    fake = buffers.Buffers(w, planes, [], [], [], [])
    gc.check_retrieve(fake, chunks_np=host_copies)
    del planes, pinned
    torch.cuda.empty_cache()


def test_llama70b_full_buffer_as_one_call():
    """The 100% buffer: the whole 40 GiB batch (4 requests x 32,768 tokens, 512 chunks,
    1,310,720 pieces of 32 KiB over 160 planes) in ONE call, in the launch configuration
    the benchmark times (after kvs_query_bw, flags 0, a side stream); every element of
    every plane against the oracle, one plane at a time."""
    s = torch.cuda.Stream()
    kvs.kvs_query_bw(s, 1 << 30)
    w = synth.llama70b()
    buf = buffers.allocate(w)
    assert buf.payload_bytes == 40 << 30
    assert sum(len(r.chunks) for r in buf.requests) * 2 * w.geom.layers * 16 == 1_310_720
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, s, 0)
    s.synchronize()
    assert kvs.kvs_check_errors(s) == kvs.KVS_OK
    gc.check_retrieve(buf)
    gc.free(buf)
