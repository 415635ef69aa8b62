"""Retrieval straight from the fast tier's pinned arena (kvs_tier_* + kvs_retrieve),
against the CPU oracle run on the objects' original bytes."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2609_35065_gb300 import kvs, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    yield


def test_claims_staged_into_the_arena_retrieve_exactly():
    g = synth.Geometry(4, 8, 128, 2, 16, 256)
    elems = 2 * g.layers * g.chunk_tokens * g.row_elems
    nbytes = elems * 2
    rng = np.random.default_rng(21)
    backing = {k: rng.integers(0, 0x7F80, size=elems, dtype=np.uint16) for k in range(10)}   # the "SSD"
    tier = kvs.Tier(capacity_objects=6, budget_objects=4, object_bytes=nbytes, arena=True)
    nb = 160
    perm = rng.permutation(nb).astype(np.int32)
    manifests = {1: [0, 1, 2], 2: [0, 3]}              # request 2 shares object 0 (a common prefix)
    tables = {1: perm[:48], 2: np.concatenate([perm[:16], perm[48:64]]).astype(np.int32)}
    planes = torch.full((2 * g.layers, nb * g.block_size * g.row_elems), synth.SENTINEL_BF16,
                        dtype=torch.int16, device="cuda")
    ptrs = [int(planes[p].data_ptr()) for p in range(planes.shape[0])]

    def stage(keys, now):
        for k in keys:
            slot = tier.object(k)["slot"]
            ctypes.memmove(tier.slot_address(slot), backing[k].ctypes.data, nbytes)
            tier.staged(k, now)

    def retrieve(claims, now):
        reqs = []
        for c in claims:
            slots = tier.begin_retrieval(c, now, len(manifests[c]))
            reqs.append(kvs.RequestArg(tables[c], [kvs.ChunkArg(tier.slot_address(s), g.chunk_tokens)
                                                   for s in slots]))
        kvs.kvs_retrieve(g, ptrs, nb, reqs, None, kvs.KVS_F_VALIDATE)
        torch.cuda.synchronize()
        for c in claims:
            tier.end_retrieval(c, now + 0.5)

    stage(tier.commit(1, manifests[1], 0.0), 0.25)
    assert tier.commit(2, manifests[2], 0.5) == [3]     # object 0 is coalesced
    stage([3], 1.5)
    retrieve([1, 2], 2.0)
    expected = [np.full(planes.shape[1], synth.SENTINEL_BF16, dtype=np.uint16) for _ in range(2 * g.layers)]
    for c in (1, 2):
        assert oracle.retrieve(g.layers, g.kv_heads, g.head_dim, g.block_size, expected, nb, 0,
                               [backing[k] for k in manifests[c]], tables[c]) == 0
    got = planes.cpu().numpy().view(np.uint16)
    for p in range(2 * g.layers):
        assert np.array_equal(got[p], expected[p]), p

    # a later claim needs two new objects: the least recently used unprotected ones are
    # evicted, their slots refilled, and retrieval again matches the oracle
    manifests[3] = [4, 5]
    tables[3] = perm[64:96]
    staged = tier.commit(3, manifests[3], 3.0)
    assert staged == [4, 5] and tier.stats(3.0)["evictions"] == 0     # two free slots left
    manifests[4] = [6, 7]
    tables[4] = perm[96:128]
    stage(staged, 3.5)
    retrieve([3], 4.0)
    staged = tier.commit(4, manifests[4], 5.0)
    assert tier.stats(5.0)["evictions"] == 2
    stage(staged, 5.5)
    retrieve([4], 6.0)
    for c in (3, 4):
        assert oracle.retrieve(g.layers, g.kv_heads, g.head_dim, g.block_size, expected, nb, 0,
                               [backing[k] for k in manifests[c]], tables[c]) == 0
    got = planes.cpu().numpy().view(np.uint16)
    for p in range(2 * g.layers):
        assert np.array_equal(got[p], expected[p]), p
    tier.close()
