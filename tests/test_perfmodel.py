"""The roofline numerator: algorithmic bytes and FLOPs per launch.

`bench.py` reports achieved = algorithmic work of one launch / its measured
duration. These tests pin that work to counts made by hand from the
definitions: each input element read once and each output written once (the
compulsory HBM traffic), and the FLOP convention of the operator (sparse
4 N b d_h; RACE 4 N r d_h + 4 N r for B, A, Num and Den; projections
4 N d_h L_s gamma for Q and K; per head).
"""
import pytest

from paper_2607_20214_gb300 import perfmodel
from paper_2607_20214_gb300.workloads import WORKLOADS


def tensor_bytes(wl, elt=None):
    """Bytes of one [B, H, N, d_h] tensor."""
    return wl.B * wl.H * wl.N * wl.d_h * (wl.elt if elt is None else elt)


@pytest.mark.parametrize("name", ["c2", "c3", "c4"])
def test_block_kernel_bytes_are_qkv_read_and_o_written(name):
    wl = WORKLOADS[name]
    w = perfmodel.kernel_work(wl, "block_attn_ws")
    assert w["bytes"] == 4 * tensor_bytes(wl)


def test_block_kernel_bytes_c3_and_c4_by_hand():
    # c3: 2 x 16 heads x 16384 x 128 bf16 = 134 217 728 bytes per tensor
    assert perfmodel.kernel_work(WORKLOADS["c3"], "block_attn_ws")["bytes"] \
        == 4 * 134_217_728
    # c4: 1 x 32 heads x 65536 x 128 bf16 = 536 870 912 bytes per tensor
    assert perfmodel.kernel_work(WORKLOADS["c4"], "block_attn_ws")["bytes"] \
        == 4 * 536_870_912


@pytest.mark.parametrize("name", ["c2", "c3", "c4"])
def test_key_side_and_hash_read_two_tensors(name):
    wl = WORKLOADS[name]
    assert perfmodel.kernel_work(wl, "race_keys_ws")["bytes"] == \
        2 * tensor_bytes(wl)  # K and V
    assert perfmodel.kernel_work(wl, "sort_hash")["bytes"] == \
        2 * tensor_bytes(wl)  # Q and K


@pytest.mark.parametrize("name", ["c2", "c3", "c4"])
def test_forward_flops_split_over_the_two_kernels(name):
    """The query-side kernel and the key-side kernel together carry the
    operator's tensor FLOPs exactly once."""
    wl = WORKLOADS[name]
    N, b, d, r = wl.N, wl.block, wl.d_h, wl.r
    Lg = wl.race_tables * wl.race_bits
    per_head = 4 * N * b * d + 4 * N * r * d + 4 * N * r + 4 * N * d * Lg
    total = (perfmodel.kernel_work(wl, "block_attn_ws")["flops"] +
             perfmodel.kernel_work(wl, "race_keys_ws")["flops"])
    assert total == wl.heads * per_head


def test_backward_tc_bytes_c5():
    """Tensor-core backward block kernel: reads Q, K, V, dO (bf16) and
    writes dQ, dK, dV (fp32) once."""
    wl = WORKLOADS["c5"]
    w = perfmodel.kernel_work(wl, "bwd_block_tc")
    assert w["bytes"] == 4 * tensor_bytes(wl) + 3 * tensor_bytes(wl, 4)
    assert w["unit"] == "tensor"


def test_roofline_picks_the_slower_resource():
    peaks = {"hbm_gbs": 1000.0, "bf16_tflops": 100.0}
    # 1 GB and 1 TFLOP: 1 ms of HBM, 10 ms of tensor time -> tensor-bound
    w = {"bytes": 1e9, "flops": 1e12, "unit": "tensor"}
    rf = perfmodel.roofline(w, 0.02, peaks)
    assert rf["bound"] == "tensor" and rf["unit"] == "TFLOP/s"
    assert rf["achieved"] == pytest.approx(50.0)
    assert rf["frac"] == pytest.approx(0.5)
    # 1 GB and 1 GFLOP: HBM-bound; 1 GB in 2 ms = 500 GB/s
    w = {"bytes": 1e9, "flops": 1e9, "unit": "tensor"}
    rf = perfmodel.roofline(w, 0.002, peaks)
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s"
    assert rf["achieved"] == pytest.approx(500.0)
    assert rf["frac"] == pytest.approx(0.5)
