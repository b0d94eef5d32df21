"""Block attention for key blocks of 256 on CTA pairs (k_block_attn_pair,
bf16, d_h = 128, gamma = 4) against the fp64 oracle.

The pair kernel takes a block's two 128-query tiles on two SMs with
cta_group::2 MMAs; each cluster walks a contiguous range of blocks, so the
cases below give clusters several blocks with head changes inside their
ranges (planes and summaries reloaded per head), both TMEM slots, and RACE
ranks below, at and above 128 (one or two feature parts). Sort orders must
match exactly; O within max-abs 2e-2 with the relative error reported.
"""
import numpy as np
import pytest
import torch

from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import Workload, make_gates_lambda, \
    make_inputs
from test_parity_gpu import compare, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def pair_wl(**kw):
    base = dict(name="pair", B=1, H=16, N=4096, d_h=128, dtype="bf16",
                block=256, race_tables=16, recipe="plain", temperature=2.0,
                seed=61, plane_seed=1061)
    base.update(kw)
    return Workload(**base)


def test_pair_kernel_runs_for_blocks_of_256():
    wl = pair_wl(H=2, N=1024)
    x = make_inputs(wl)
    elsaa.elsaa_profile_start()
    g = run_gpu(wl, x)
    prof = elsaa.elsaa_profile_stop()
    assert "block_attn_pair" in prof and "block_attn_ws" not in prof, prof
    compare(wl, g, run_oracle(wl, x), label="pair small")


@pytest.mark.parametrize("L", [4, 8, 12, 16])
def test_pair_several_blocks_per_cluster(L):
    """16 heads of 16 blocks: 256 blocks over the clusters, 3-4 each, so
    ranges cross head boundaries; r = 16 L (64 .. 256)."""
    wl = pair_wl(race_tables=L, seed=62 + L)
    x = make_inputs(wl)
    g = run_gpu(wl, x)
    heads = [(0, 0), (0, 5), (0, 15)]
    compare(wl, g, run_oracle(wl, x, heads=heads), label="pair L=%d" % L)


def test_pair_batches_gates_lambda_and_fp32_output():
    wl = pair_wl(B=2, H=8, N=2048, seed=71)
    x = make_inputs(wl)
    gates, lam = make_gates_lambda(wl, seed=13)
    ref = run_oracle(wl, x, gates=gates, lam=lam, heads=[(0, 3), (1, 7)])
    g32 = run_gpu(wl, x, gates=gates, lam=lam, out_fp32=1)
    assert g32["O_raw"].dtype == torch.float32
    compare(wl, g32, ref, label="pair gates fp32")
    g16 = run_gpu(wl, x, gates=gates, lam=lam)
    assert torch.equal(g16["O_raw"], g32["O_raw"].to(torch.bfloat16))


def test_pair_one_block_per_cluster_and_duplicate_keys():
    """Fewer blocks than clusters (one block each: one slot idle) and the
    duplicated-key recipe (runs of equal codes across block edges)."""
    wl = pair_wl(H=2, N=512, recipe="dup_keys", seed=72)
    x = make_inputs(wl)
    compare(wl, run_gpu(wl, x), run_oracle(wl, x), label="pair dup")


def test_pair_rows_of_a_large_head():
    """N = 16384 (64 blocks per head, 4 heads): sampled rows of two heads,
    the last rows included."""
    wl = pair_wl(H=4, N=16384, seed=73)
    x = make_inputs(wl)
    rows = np.unique(np.concatenate([
        np.random.default_rng(5).choice(wl.N, 400, replace=False),
        np.arange(wl.N - 300, wl.N)]))
    g = run_gpu(wl, x)
    compare(wl, g, run_oracle(wl, x, heads=[(0, 1), (0, 3)], rows=rows),
            label="pair N=16384")


@pytest.mark.parametrize("over", [dict(fusion_mode=1), dict(beta=4.0),
                                  dict(lam=0.25), dict(eps=1e-2),
                                  dict(sort_bits=0)])
def test_pair_parameter_variants(over):
    """Fusion mode, RACE temperature, lambda, epsilon and the identity
    order (no sort bits: every block is a run of consecutive tokens)."""
    wl = pair_wl(H=4, N=2048, seed=74).with_(**over)
    x = make_inputs(wl)
    compare(wl, run_gpu(wl, x), run_oracle(wl, x, heads=[(0, 0), (0, 3)]),
            label=str(over))
