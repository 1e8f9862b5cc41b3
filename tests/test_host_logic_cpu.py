"""Host-side integer logic of the kernels, checked exhaustively on the CPU."""
import numpy as np


def test_cube_index_reciprocal_division_is_exact():
    """The sparse kernel finds a cube's coordinates as floor((a + 0.5) * fl(1/d)) in fp32 instead of
    an integer division a / d.  That equals a / d for every block id a and divisor d the library
    accepts (at most 7008 blocks), checked here for all pairs in fp32 arithmetic."""
    a = np.arange(7008, dtype=np.int64)
    af = a.astype(np.float32) + np.float32(0.5)
    for d in range(1, 7009):
        r = np.float32(1.0 / d)                       # the host's fp64 reciprocal rounded to fp32
        q = np.floor(af * r).astype(np.int64)         # fp32 product, truncated
        assert np.array_equal(q, a // d), d
