"""The CPU oracle against facts that do not come from itself (runs without a GPU)."""
import numpy as np
import pytest

import oracle
import oracle_pins as pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(oracle_lib, pin):
    pin(oracle_lib)


def test_bounds_status_and_partial_write(oracle_lib):
    """A block id outside [0, NB) or a too-short block table is reported (-2) and only
    the elements of the offending tokens are skipped."""
    L, H, D, B, nb = 1, 1, 2, 2, 4
    planes = [np.zeros(nb * B * H * D, np.uint16) for _ in range(2 * L)]
    chunk = np.arange(1, 2 * L * 6 * H * D + 1, dtype=np.uint16)
    rc = oracle.retrieve(L, H, D, B, planes, nb, 0, [chunk], np.array([1, 4, 0], np.int32),
                         lib=oracle_lib)
    assert rc == -2
    k = planes[0].reshape(nb * B, H * D)
    # tokens 0,1 -> block 1; tokens 2,3 -> block 4 (invalid, skipped); tokens 4,5 -> block 0
    assert k[2:4].tolist() == [[1, 2], [3, 4]]
    assert k[0:2].tolist() == [[9, 10], [11, 12]]
    assert np.all(k[4:] == 0)
    rc = oracle.retrieve(L, H, D, B, planes, nb, 0, [chunk], np.array([1, 2], np.int32),
                         lib=oracle_lib)
    assert rc == -2                                     # table covers 4 of 6 tokens


def test_plane_range_restriction(oracle_lib):
    """Only planes [p0, p1) are written; the others may even be absent."""
    L, H, D, B, nb = 3, 2, 4, 4, 8
    full = [np.zeros(nb * B * H * D, np.uint16) for _ in range(2 * L)]
    part = [None] * (2 * L)
    part[2] = np.zeros_like(full[2]); part[3] = np.zeros_like(full[3])
    chunk = np.arange(1, 2 * L * 8 * H * D + 1, dtype=np.uint16)
    bt = np.array([5, 1], np.int32)
    assert oracle.retrieve(L, H, D, B, full, nb, 0, [chunk], bt, lib=oracle_lib) == 0
    assert oracle.retrieve(L, H, D, B, part, nb, 0, [chunk], bt, p0=2, p1=4, lib=oracle_lib) == 0
    assert np.array_equal(part[2], full[2]) and np.array_equal(part[3], full[3])


def test_fill(oracle_lib):
    a = np.zeros(7, np.uint16)
    oracle.fill(a, 0x7FA5)
    assert np.all(a == 0x7FA5)
