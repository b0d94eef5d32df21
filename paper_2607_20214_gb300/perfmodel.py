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
    if getattr(wl, "causal", 0):
        return causal_flop_model(wl)
    b = keys_per_query(wl)
    per_head = (4 * N * b * d + 4 * N * r * d + 4 * N * r
                + 4 * N * d * wl.race_tables * wl.race_bits)
    heads = wl.heads
    return {
        "tensor_flops": per_head * heads,
        "sparse_flops": 4 * N * b * d * heads,
        "hash_flops": 4 * N * d * wl.sort_bits * heads,
        "bytes": 4 * N * d * wl.elt * heads,
    }


# CUDA-core fp32 peak of a 152-SM GB300 at its 2070 MHz maximum clock:
# 152 SMs x 128 FP32 lanes x 2 FLOP per FMA x 2.07e9 / s.
SIMT_FP32_PEAK_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def causal_levels(wl: Workload):
    """(levels, base segment length) of the unrolled CausalSparse
    recursion: halve N until a segment fits the base length N_0."""
    n, lv = wl.N, 0
    while n > wl.causal_base_len:
        n //= 2
        lv += 1
    return lv, n


def causal_flop_model(wl: Workload) -> dict:
    """Useful tensor FLOPs of Algorithm "Causal ELSAA", per head:
    base segments 4 d_h sum_i (i + 1) over each segment (exact causal
    attention, ~2 N n_leaf d_h); each level's SortLSH blocks 4 (N / 2) b d_h;
    causal RACE: chunk summaries 2 N r d_h + 2 N r, inter-chunk readout
    2 N r d_h + 2 N r, intra-chunk masked products (C + 1) / 2 keys per row
    of 2 (r + d_h) each (C = 128 on the device), projections 4 N d_h L_s
    gamma. Bytes: Q, K, V read once and O written once."""
    N, b, d, r = wl.N, wl.block, wl.d_h, wl.r
    lv, n_leaf = causal_levels(wl)
    C = 128
    sparse = 2 * d * N * (n_leaf + 1) + lv * 4 * (N // 2) * b * d
    race = (4 * N * r * d + 4 * N * r + N * (C + 1) * (r + d)
            + 4 * N * d * wl.race_tables * wl.race_bits)
    heads = wl.heads
    return {"tensor_flops": (sparse + race) * heads,
            "sparse_flops": sparse * heads,
            "hash_flops": 4 * N * d * wl.sort_bits * heads,
            "bytes": 4 * N * d * wl.elt * heads}


def backward_flop_model(wl: Workload) -> dict:
    """Tensor FLOPs and algorithmic HBM bytes of one backward pass (dQ, dK,
    dV in fp32), per head: sparse blocks 10 N b d_h (recomputed scores, P V
    for O_s, and the products for dV, dP, dQ, dK), RACE 8 N r d_h (Num
    recomputed, gB and gA sums, dL/dphi of queries and keys, dV of the
    summaries), projections 8 N d_h L_s gamma (recomputed and
    back-propagated for queries and keys). Bytes: Q, K, V and dO read once,
    dQ, dK, dV written once in fp32."""
    N, b, d, r = wl.N, keys_per_query(wl), wl.d_h, wl.r
    per_head = (10 * N * b * d + 8 * N * r * d
                + 8 * N * d * wl.race_tables * wl.race_bits)
    return {"tensor_flops": per_head * wl.heads,
            "bytes": (4 * N * d * wl.elt + 3 * N * d * 4) * wl.heads}


def keys_per_query(wl: Workload) -> int:
    """Keys each query attends to in the sparse branch: its block and the
    neighbouring sorted blocks, (2 r + 1) b (Section 5), at most N (the
    clipped windows at the two ends are counted as full). With the top-k
    selector the tensor cores score all c b candidate keys of a query
    block (the unselected ones are masked)."""
    if getattr(wl, "selector", 0) == 1:
        return min(wl.N, wl.topk_blocks * wl.block)
    return min(wl.N, (2 * getattr(wl, "neighbor_blocks", 0) + 1) * wl.block)


def kernel_work(wl: Workload, kernel: str) -> dict:
    """Algorithmic work of ONE launch of a kernel over the whole workload.

    bytes: compulsory HBM traffic (each input element read once, each output
    written once); flops: the kernel's share of the operator's arithmetic;
    unit: which engine runs that arithmetic ("tensor" or "alu").
    """
    N, b, d, r = wl.N, keys_per_query(wl), wl.d_h, wl.r
    H = wl.heads
    Lg = wl.race_tables * wl.race_bits
    e = wl.elt
    simt = kernel.endswith("_simt") or wl.dtype == "fp32"
    if kernel.startswith("block_attn"):
        by = H * 4 * N * d * e
        fl = H * (4 * N * b * d + 2 * N * r * d + 2 * N * r + 2 * N * d * Lg)
    elif kernel.startswith(("race_partial", "race_keys")):
        by = H * 2 * N * d * e
        fl = H * (2 * N * r * d + 2 * N * r + 2 * N * d * Lg)
    elif kernel.startswith("bwd_block"):
        # recompute scores and O_s, dZ, dV, dK, dQ (12 N b d) and the query
        # side of RACE (4 N r d + 4 N d Lg); reads Q, K, V, dO, writes dQ,
        # dK, dV in fp32. The CUDA-core kernel also writes gNum (fp32) for
        # a separate pass; the tensor-core kernel sums gB, gA itself
        # (2 N r (d + 1)) on the tensor cores.
        tc = kernel.endswith("_tc")
        by = H * (4 * N * d * e + (3 if tc else 4) * N * d * 4)
        fl = H * (12 * N * b * d + 4 * N * r * d + 4 * N * d * Lg +
                  (2 * N * r * (d + 1) if tc else 0))
        simt = not tc
    elif kernel.startswith("bwd_keys"):
        # reads K, V, adds into dK, dV (fp32 read + write); the tensor-core
        # kernel also reads the block kernel's gB, gA partials (about 1 %)
        by = H * (2 * N * d * e + 4 * N * d * 4)
        fl = H * (4 * N * r * d + 4 * N * d * Lg)
        simt = not kernel.endswith("_tc")
    elif kernel.startswith("causal_attn_base"):
        # exact causal attention of the base segments: reads Q, K, V once,
        # writes the running O (fp32) and log d
        _, n_leaf = causal_levels(wl)
        by = H * (3 * N * d * e + N * d * 4 + N * 4)
        fl = H * 2 * d * N * (n_leaf + 1)
        simt = False
    elif kernel.startswith("causal_attn_merge"):
        # one level's SortLSH blocks: half the rows as queries, half as
        # keys and values; the running O and log d read and written
        by = H * (3 * (N // 2) * d * e + (N // 2) * (d + 1) * 4 * 2)
        fl = H * 4 * (N // 2) * wl.block * d
        simt = False
    elif kernel.startswith("causal_race"):
        # reads Q, K, V, the chunk's prefix state sB (bf16) and the sparse
        # result, writes O; inter + intra products and projections
        nc = N // 128
        by = H * (3 * N * d * e + nc * r * d * 2 + N * (d + 1) * 4 +
                  N * d * e)
        fl = H * (2 * N * r * d + N * 129 * (r + d) +
                  4 * N * d * Lg)
        simt = False
    elif kernel.startswith("causal_scan"):
        # prefix states chunk after chunk: reads K, V again, writes sB_n
        # (bf16) and sA_n of every 128-key chunk; the chunk summaries
        # phi^T [V | 1] and the projections on the tensor cores
        nc = N // 128
        by = H * (2 * N * d * e + nc * r * (d * 2 + 4))
        fl = H * (2 * N * r * (d + 16) + 2 * N * d * Lg)
        simt = False
    elif kernel.startswith("bwd_race_sums"):
        by = H * (N * d * e + N * d * 4)
        fl = H * (2 * N * r * d + 2 * N * r + 2 * N * d * Lg)
        simt = True
    elif kernel.startswith("prep_planes"):
        lg = wl.race_tables * wl.race_bits
        by = wl.H * lg * d * 4 + wl.H * ((lg + 15) // 16 * 16) * d * 2
        fl = 0
        simt = True
    elif kernel.startswith("race_reduce"):
        by = H * r * (d + 1) * 4  # the summaries A and B, written once
        fl = 0
        simt = True
    elif kernel.startswith("topk_select"):
        # block sums (Q and K read through the sort orders), block scores,
        # and per query the canonical fp32 chains over the c b candidate
        # keys (each query block stages its candidates once): reads Q once
        # and the candidate keys c times, writes the bitmask
        c = getattr(wl, "topk_blocks", 1)
        by = H * (2 * N * d * e + N * d * e + c * N * d * e + N * c * wl.block
                  // 8)
        fl = H * (2 * N * c * wl.block * d + 2 * (N // wl.block) ** 2 * d)
        simt = True
    elif kernel.startswith("sort_hash"):
        by = H * 2 * N * d * e
        fl = H * 4 * N * d * wl.sort_bits
        simt = True
    else:
        by = H * N * 8
        fl = 0
        simt = True
    return {"bytes": by, "flops": fl, "unit": "alu" if simt else "tensor"}


def roofline(work: dict, seconds: float, peaks: dict) -> dict:
    """Bound, achieved and peak of one launch taking `seconds`."""
    hbm = peaks["hbm_gbs"]
    if work["unit"] == "tensor":
        fpk = peaks["bf16_tflops"]
    else:
        fpk = SIMT_FP32_PEAK_TFLOPS
    t_bytes = work["bytes"] / (hbm * 1e9)
    t_flops = work["flops"] / (fpk * 1e12) if work["flops"] else 0.0
    if t_bytes >= t_flops:
        ach = work["bytes"] / seconds / 1e9
        return {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                "frac": ach / hbm}
    ach = work["flops"] / seconds / 1e12
    return {"bound": work["unit"], "achieved": ach, "peak": fpk,
            "unit": "TFLOP/s", "frac": ach / fpk}
