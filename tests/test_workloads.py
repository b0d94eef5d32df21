"""The seeded input recipes (CPU): determinism, shapes and planted structure."""
import torch

from paper_2607_20214_gb300.workloads import (WORKLOADS, make_inputs,
                                              head_temperatures)


def test_deterministic_and_shapes():
    wl = WORKLOADS["c1"]
    a = make_inputs(wl)
    b = make_inputs(wl)
    for key in ("q", "k", "v", "w_sort", "w_race"):
        assert torch.equal(a[key], b[key])
    assert a["q"].shape == (1, 1, 1024, 64) and a["q"].dtype == torch.float32
    assert a["w_sort"].shape == (1, 5, 64)
    assert a["w_race"].shape == (1, 4, 4, 64)
    # RACE planes hold bf16-representable values
    assert torch.equal(a["w_race"], a["w_race"].bfloat16().float())


def test_planted_heads_hold_near_copies_of_needle_queries():
    wl = WORKLOADS["c2"].with_(B=1, H=4, N=512)
    x = make_inputs(wl)
    temps = head_temperatures(wl)
    assert x["k"].dtype == torch.bfloat16
    q_raw = x["q"].float() / temps.view(1, -1, 1, 1)
    for h in range(4):
        k = x["k"][0, h].float()
        needles = q_raw[0, h, ::8]
        dist = torch.cdist(k, needles).min(dim=1).values
        if h % 2 == 0:  # planted: every key within the 0.1 noise of a needle
            assert dist.max() < 0.1 * 8 * 2
        else:
            assert dist.min() > 2.0


def test_duplicate_keys_recipe():
    wl = WORKLOADS["c4"].with_(H=2, N=1024)
    x = make_inputs(wl)
    k = x["k"]
    m = torch.arange(1024 // 128) * 64
    assert torch.equal(k[:, :, 512 + m], k[:, :, m])


def test_training_workload_has_upstream_gradient():
    wl = WORKLOADS["c5"].with_(B=1, H=2, N=256)
    x = make_inputs(wl)
    assert x["do"].shape == x["q"].shape
