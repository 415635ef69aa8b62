"""kvs_retrieve_noalloc against kvs_retrieve.

kvs_retrieve_noalloc serves callers that cannot let a library allocate GPU
memory: serving runtimes that reserve nearly all free HBM for their own KV
block pool and sub-allocate it themselves, and latency-critical paths where a
cudaMalloc / cudaFree would synchronise the device.  Its scratch is a static
device array compiled into the library.  Here two calls in a row must give
exactly the bytes kvs_retrieve gives (the path only copies bytes, so the
tolerance is zero), and free device memory must not shrink during a call.
"""
import numpy as np
import pytest
import torch

from paper_2609_35065_gb300 import buffers, kvs, synth

pytestmark = pytest.mark.gpu


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
    return buf.planes, other, free_before, free_after


def test_noalloc_matches_kvs_retrieve_on_two_calls_in_a_row():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    for k, w in enumerate([synth.tiny(), _mixed_shared_workload()]):
        want, got, free_before, free_after = _both_paths(w)
        assert torch.equal(want, got), f"call {k + 1}: kvs_retrieve_noalloc differs from kvs_retrieve"
        assert not torch.all(got == got.view(-1)[0]), "nothing was written"
        if k == 1:
            # the scratch array was set up on the first call; this call allocates nothing
            assert free_after >= free_before, (free_before, free_after)


def test_noalloc_refuses_calls_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    # 4096-token chunks of 1-token blocks: 16 KiB of block ids per chunk, 80 chunks > 1 MiB
    fake = 1 << 20
    g = (1, 1, 8, 2, 1, 4096)
    chunks = [kvs.ChunkArg(fake + 65536 * j, 4096) for j in range(80)]
    req = kvs.RequestArg(np.arange(80 * 4096, dtype=np.int32), chunks)
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_noalloc(g, [fake, fake], 80 * 4096, [req], None, 0)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
    assert "KVS_NOALLOC_SCRATCH_BYTES" in str(ei.value)
    with pytest.raises(kvs.KvsError) as ei:
        kvs.kvs_retrieve_noalloc(g, [fake, fake], 80 * 4096, [req], None, kvs.KVS_F_FORCE_HBMCOPY)
    assert ei.value.code == kvs.KVS_ERR_UNSUPPORTED
