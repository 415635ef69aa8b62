"""Library state through its lifetime: launch accounting, shutdown, re-initialisation."""
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


def _retrieve(buf, flags=0):
    w = buf.workload
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, buf.requests, None, flags)


def test_one_launch_per_source_class_and_none_for_an_empty_call():
    buf = buffers.allocate(synth.tiny())
    w = buf.workload
    n0 = kvs.kvs_stat_launches()
    _retrieve(buf, kvs.KVS_F_FORCE_HOSTLINK)              # host chunks, host-link kernel: one launch
    torch.cuda.synchronize()
    assert kvs.kvs_stat_launches() == n0 + 1
    kvs.kvs_retrieve(w.geom, buf.plane_ptrs, w.num_blocks, [], None, 0)
    assert kvs.kvs_stat_launches() == n0 + 1
    gc.check_retrieve(buf)


def test_shutdown_releases_state_and_the_next_call_starts_afresh():
    rep = kvs.kvs_query_bw(None, 64 << 20)
    assert rep["hostlink_ctas"] >= 0
    buf = buffers.allocate(synth.tiny(), store=True)
    _retrieve(buf, kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    assert kvs.kvs_shutdown() == kvs.KVS_OK
    # the defaults are back until the next probe
    got = kvs.kvs_get_choice()
    assert got["chosen_retrieve_host"] == kvs.KVS_VARIANT_HOSTLINK
    assert got["chosen_kernel_device"] == kvs.KVS_KERNEL_LDG
    assert got["probe_bytes"] == 0
    # a fresh state gives the same exact result
    buf.planes.fill_(int(torch.tensor([synth.SENTINEL_BF16], dtype=torch.int32).to(torch.int16)))
    torch.cuda.synchronize()
    _retrieve(buf, kvs.KVS_F_VALIDATE)
    w = buf.workload
    kvs.kvs_store(w.geom, buf.plane_ptrs, w.num_blocks, buf.store_requests, None, kvs.KVS_F_VALIDATE)
    torch.cuda.synchronize()
    gc.check_retrieve(buf)
    gc.check_store(buf)
    assert kvs.kvs_check_errors(None) == kvs.KVS_OK
