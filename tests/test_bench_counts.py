"""The candidate counts behind bench.py's throughput and roofline figures, checked by
brute-force enumeration on small sizes (CPU only)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def _apx_rec_candidates(p, s):
    # eq. apx_rec with 0-based unique values: layer i = 3..s, output j in [i-1, p-1],
    # predecessor k in [i-2, j-1] (k < j, at least i-2 values before k)
    return sum(1 for i in range(3, s + 1) for j in range(i - 1, p) for k in range(i - 2, j))


@pytest.mark.parametrize("p,s", [(1, 4), (2, 3), (5, 3), (7, 8), (16, 5), (40, 9), (64, 16)])
def test_candidates_per_multiplier_is_the_recurrence_count(p, s):
    import bench
    assert bench.candidates_per_multiplier(p, s) == _apx_rec_candidates(p, s)


def _opt_candidates(n, s, nL):
    # Sec. 4 layers i = 3..s over states (k, l) -> (l, j), k < l < j; at i = 3 the
    # predecessor k is a first-value candidate (k < nL), above it k >= i - 3
    c = 0
    for i in range(3, s + 1):
        for l in range(n - 1):
            ks = [k for k in range(l) if (k < nL if i == 3 else k >= i - 3)]
            c += len(ks) * (n - 1 - l)
    return c


@pytest.mark.parametrize("n,s,nL", [(6, 3, 1), (10, 5, 1), (12, 6, 3), (20, 8, 2)])
def test_opt_candidates_is_the_recurrence_count(n, s, nL):
    import bench
    assert bench.opt_candidates(n, s, 1, nL) == _opt_candidates(n, s, nL)
    assert bench.opt_candidates(n, s, 3, nL) == 3 * _opt_candidates(n, s, nL)


@pytest.mark.parametrize("p,s,G", [(64, 16, 8), (130, 5, 7), (131072, 16, 43)])
def test_executed_candidates_counts_tile_units_and_diagonal_triangles(p, s, G):
    """bench.py's executed count: every 64 x 64 off-diagonal tile unit the kernel ran,
    over the s - 2 layers, plus one 64-column triangle (pairs k < j) per column block
    and multiplier."""
    import bench
    L = s - 2
    blocks = -(-p // 64)
    tri = sum(1 for j in range(64) for k in range(j))
    assert bench.executed_candidates({"tiles_run": 0}, p, s, G) == G * blocks * tri * L
    assert (bench.executed_candidates({"tiles_run": 5}, p, s, G)
            - bench.executed_candidates({"tiles_run": 0}, p, s, G)) == 5 * 64 * 64 * L
