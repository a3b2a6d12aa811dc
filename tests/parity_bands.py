"""Comparison bands shared by the acceptance parity tests.

The acceptance decisions are bit-exact against the fp64 oracle except inside
two narrow bands where fp32 and fp64 may legitimately decide differently:
* an accept test with |u_i - p_i(x_i)/q_i(x_i)| < 1e-5 (the band the
  acceptance rule's tolerance names);
* a final draw with u_k within 1e-6 of either CDF value that brackets the
  drawn token (the kernels' fp32 running sums resolve the CDF to ~1e-8).
Requests in a band are counted; they must stay rare, so that a kernel that
drifts into the bands still fails: at most 1% of the requests (at least 2
allowed, for small samples).  With uniform u the expected rate is about
2e-5 per accept test, far below that bound.
"""
import math

NEAR_TIE = 1e-5
DRAW_TIE = 1e-6


def max_near_ties(n_requests: int) -> int:
    return max(2, math.ceil(0.01 * n_requests))


def check_tie_rate(n_ties: int, n_requests: int, what: str = "") -> None:
    assert n_ties <= max_near_ties(n_requests), (
        f"{what}: {n_ties} of {n_requests} requests fall in a near-tie band "
        f"(at most {max_near_ties(n_requests)} allowed)")
