"""Work and traffic model of the operator, used by the benchmark.

Counts follow the paper's complexity analysis (Section 6 and the numerical
example of Appendix F) plus the tensor-core FLOP convention of the benchmark.
"""
from __future__ import annotations

from .workloads import Workload


def interaction_counts(N: int, s: int, L_s: int, gamma: int) -> dict:
    """Attention interaction counts per head (Section 6 complexity model).

    full = N^2, sparse = N s, race = N L_s 2^gamma, elsaa = sparse + race.
    """
    full = N * N
    sparse = N * s
    race = N * L_s * (1 << gamma)
    return {"full": full, "sparse": sparse, "race": race,
            "elsaa": sparse + race}


def flop_model(wl: Workload) -> dict:
    """Tensor FLOPs and algorithmic HBM bytes of one forward pass.

    Per head: sparse blocks 4 N b d_h (scores and P V), RACE 4 N r d_h + 4 N r
    (key summaries B and A, query readout Num and Den), RACE projections
    4 N d_h L_s gamma (queries and keys). Algorithmic bytes read Q, K, V once
    and write O once. The sort hash (4 N d_h n_s CUDA-core FLOPs) is reported
    separately.
    """
    N, b, d, r = wl.N, wl.block, wl.d_h, wl.r
    per_head = (4 * N * b * d + 4 * N * r * d + 4 * N * r
                + 4 * N * d * wl.race_tables * wl.race_bits)
    heads = wl.heads
    return {
        "tensor_flops": per_head * heads,
        "sparse_flops": 4 * N * b * d * heads,
        "hash_flops": 4 * N * d * wl.sort_bits * heads,
        "bytes": 4 * N * d * wl.elt * heads,
    }
