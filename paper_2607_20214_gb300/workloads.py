"""Seeded synthetic workloads for the ELSAA attention operator.

This module is the one piece shared by the CUDA path's callers (tests, bench,
smoke) and the CPU oracle's callers: it draws Q, K, V, the hash planes and the
upstream gradient from fixed seeds. It holds none of the operator's arithmetic
(no hashing, sorting, attention, RACE features or fusion); it only generates
tensors with the shapes and value distributions of the five workloads.

Shapes follow the paper's problem statement (Section 3: one head has
Q, K, V in R^{N x d_h}; multi-head applies the operator per head), laid out
as [B, H, N, d_h]. Hyper-parameter defaults follow Table 7 (attention
hyper-parameters): RACE hash bits gamma = 4, sortLSH bits = 5,
epsilon = 1e-6; lambda = 1 is the initial value of the learned scalar
(Appendix D, experiment hyperparameters).
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import torch


@dataclass(frozen=True)
class Workload:
    """One problem instance of the operator (all heads of one batch)."""

    name: str
    B: int
    H: int
    N: int
    d_h: int
    dtype: str  # "fp32" or "bf16": type of Q, K, V and O
    block: int  # sortLSH block size b (each query attends to exactly b keys)
    race_tables: int  # L_s
    race_bits: int = 4  # gamma, so R = 2**gamma buckets per table
    sort_bits: int = 5  # bits of the angular sort hash
    gray_order: int = 1  # 1: sort by rank in the reflected Gray sequence
    beta: float = 1.0
    eps: float = 1e-6
    lam: float = 1.0
    fusion_mode: int = 0  # 0: ELSAA multiplier, 1: Sort_Lsh_RACE ablation (m = 1)
    causal: int = 0  # 1: Algorithm "Causal ELSAA"
    causal_chunk: int = 128  # C of causal RACE
    causal_base_len: int = 4096  # N_0 of CausalSparse (Table 7, text: 4096)
    neighbor_blocks: int = 0  # r neighbouring sorted key blocks per side
    selector: int = 0  # 0: sorted blocks; 1: per-query top-k (candidates)
    topk: int = 0  # k keys per query with selector 1
    topk_blocks: int = 1  # c candidate key blocks per query block
    recipe: str = "plain"  # input recipe, see make_inputs
    temperature: float = 1.0
    seed: int = 0
    plane_seed: int = 1000
    backward: bool = False
    note: str = ""

    @property
    def r(self) -> int:
        """Total RACE bucket features S_R = L_s * 2**gamma (the low-rank rank)."""
        return self.race_tables * (1 << self.race_bits)

    @property
    def heads(self) -> int:
        return self.B * self.H

    @property
    def tokens(self) -> int:
        return self.B * self.N

    @property
    def torch_dtype(self) -> torch.dtype:
        return torch.float32 if self.dtype == "fp32" else torch.bfloat16

    @property
    def elt(self) -> int:
        return 4 if self.dtype == "fp32" else 2

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workloads. Sparse budget k is the sortLSH block size b; the
# low-rank rank r is S_R = L_s * 2**gamma with gamma = 4, so L_s = r / 16.
WORKLOADS = {
    "c1": Workload("c1", B=1, H=1, N=1024, d_h=64, dtype="fp32", block=32,
                   race_tables=4, recipe="plain", temperature=2.0, seed=0,
                   plane_seed=1001),
    "c2": Workload("c2", B=4, H=12, N=4096, d_h=64, dtype="bf16", block=64,
                   race_tables=8, recipe="planted", seed=1, plane_seed=1002),
    "c3": Workload("c3", B=2, H=16, N=16384, d_h=128, dtype="bf16", block=128,
                   race_tables=16, recipe="uniform_temp", seed=2,
                   plane_seed=1003),
    "c4": Workload("c4", B=1, H=32, N=65536, d_h=128, dtype="bf16", block=256,
                   race_tables=16, recipe="dup_keys", seed=3, plane_seed=1004),
    # c3 through Algorithm "Causal ELSAA": C = 128, N_0 = 4096 (Table 7's
    # text setting), so CausalSparse has two levels above 4096-row segments
    "c3c": Workload("c3c", B=2, H=16, N=16384, d_h=128, dtype="bf16",
                    block=128, race_tables=16, recipe="uniform_temp", seed=2,
                    plane_seed=1003, causal=1, causal_chunk=128,
                    causal_base_len=4096),
    "c5": Workload("c5", B=8, H=12, N=8192, d_h=64, dtype="bf16", block=64,
                   race_tables=8, recipe="plain", temperature=2.0, seed=4,
                   plane_seed=1005, backward=True),
}

# Temperatures of the mixed-head workload, cycled over the head index.
_CYCLE_TEMPS = (0.5, 1.0, 2.0, 4.0)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randn(shape, g, device):
    return torch.randn(*shape, generator=g, device=device, dtype=torch.float32)


def make_planes(wl: Workload, device="cpu"):
    """Hash planes, drawn per head and shared by Q and K.

    w_sort: [H, sort_bits, d_h] fp32, i.i.d. N(0, 1) (angular sort hash).
    w_race: [H, L_s, gamma, d_h] fp32 holding bf16-representable values,
            i.i.d. N(0, 1) rows as in Algorithm RACE (W^(l) with Gaussian rows).
    """
    g = _gen(wl.plane_seed, device)
    w_sort = _randn((wl.H, wl.sort_bits, wl.d_h), g, device)
    w_race = _randn((wl.H, wl.race_tables, wl.race_bits, wl.d_h), g, device)
    w_race = w_race.to(torch.bfloat16).to(torch.float32)
    return w_sort.contiguous(), w_race.contiguous()


def head_temperatures(wl: Workload, device="cpu") -> torch.Tensor:
    """Per-head query temperature T_h of the workload recipe, shape [H]."""
    if wl.recipe == "planted":
        return torch.tensor([_CYCLE_TEMPS[h % 4] for h in range(wl.H)],
                            dtype=torch.float32, device=device)
    if wl.recipe == "uniform_temp":
        g = _gen(wl.seed + 500, "cpu")
        t = torch.rand(wl.H, generator=g, dtype=torch.float32) * 3.5 + 0.5
        return t.to(device)
    return torch.full((wl.H,), float(wl.temperature), dtype=torch.float32,
                      device=device)


def make_inputs(wl: Workload, device="cpu") -> dict:
    """Draw Q, K, V (and dO for the training workload) for a workload.

    Recipes:
      plain        Q, K, V ~ N(0, 1); Q multiplied by the workload temperature.
      planted      per-head temperature cycling (0.5, 1, 2, 4). In even heads
                   every query i = 0 (mod 8) is a needle: the 8 keys
                   K[pi(i + t)], t = 0..7, are set to q_i + 0.1 N(0, 1), where
                   pi is a seeded permutation, so each key is planted once.
                   Q is scaled by the temperature after planting.
      uniform_temp per-head temperature ~ U[0.5, 4].
      dup_keys     every 64th key is repeated half a sequence later:
                   K[N/2 + 64 m] = K[64 m] for m in [0, N/128).
    Values are drawn in fp32 and then cast to the workload dtype, so both the
    CUDA path and the oracle read exactly the same (quantised) numbers.
    """
    g = _gen(wl.seed, device)
    shape = (wl.B, wl.H, wl.N, wl.d_h)
    q = _randn(shape, g, device)
    k = _randn(shape, g, device)
    v = _randn(shape, g, device)
    if wl.recipe == "planted":
        gp = _gen(wl.seed + 7, "cpu")
        n = wl.N
        for h in range(0, wl.H, 2):
            for b in range(wl.B):
                pi = torch.randperm(n, generator=gp).to(device)
                src = (torch.arange(n, device=device) // 8) * 8
                noise = _randn((n, wl.d_h), g, device)
                k[b, h, pi] = q[b, h, src] + 0.1 * noise
    if wl.recipe == "dup_keys":
        m = torch.arange(wl.N // 128, device=device) * 64
        k[:, :, wl.N // 2 + m] = k[:, :, m]
    temps = head_temperatures(wl, device)
    q = q * temps.view(1, wl.H, 1, 1)
    out = {
        "q": q.to(wl.torch_dtype).contiguous(),
        "k": k.to(wl.torch_dtype).contiguous(),
        "v": v.to(wl.torch_dtype).contiguous(),
    }
    if wl.backward:
        out["do"] = _randn(shape, g, device).to(wl.torch_dtype).contiguous()
    w_sort, w_race = make_planes(wl, device)
    out["w_sort"] = w_sort
    out["w_race"] = w_race
    return out


def make_gates_lambda(wl: Workload, seed: int, device="cpu"):
    """Per-token gates in (0, 1)^2 and per-token lambda > 0, for tests.

    Gates stand in for sigma(G_theta(q_i)) (Section 3.3); lambda_i stands in
    for c + sigma(w^T q_i + b) (Appendix D, experiment hyperparameters). Both are plain seeded draws.
    """
    g = _gen(seed, device)
    gates = torch.rand((wl.B, wl.H, wl.N, 2), generator=g, device=device,
                       dtype=torch.float32) * 0.98 + 0.01
    lam = torch.rand((wl.B, wl.H, wl.N), generator=g, device=device,
                     dtype=torch.float32) * 1.5 + 0.3
    return gates.contiguous(), lam.contiguous()


def make_gate_mlp(wl: Workload, hidden: int = 64, seed: int = 7,
                  device="cpu", w_lambda_std: float = 0.05) -> dict:
    """Parameters of the token-wise gate MLP and of the query-dependent
    lambda, per head (Section 3.3; Appendix D "gate hidden dim" 64 or 128;
    Appendix D for lambda).

    w1 [H, g, d] and w_lambda [H, d] hold bf16-representable fp32 values
    (like the RACE planes); w1 ~ N(0, 1/d), b1 ~ 0.1 N(0, 1),
    w2 [H, 2, g] ~ N(0, 1/g), b2 [H, 2] ~ 0.5 N(0, 1). lambda: c = 0.3 and
    b = 0 (so c + sigmoid(b) = 0.8, the paper's initial average target),
    w_lambda ~ w_lambda_std N(0, 1) (the paper initialises it at std 1e-3;
    tests use a larger spread so the lambda path varies), lambda_min = 1e-6.
    """
    g = _gen(seed, device)
    d = wl.d_h
    w1 = _randn((wl.H, hidden, d), g, device) / float(d) ** 0.5
    w1 = w1.to(torch.bfloat16).to(torch.float32)
    b1 = 0.1 * _randn((wl.H, hidden), g, device)
    w2 = _randn((wl.H, 2, hidden), g, device) / float(hidden) ** 0.5
    b2 = 0.5 * _randn((wl.H, 2), g, device)
    w_lambda = w_lambda_std * _randn((wl.H, d), g, device)
    w_lambda = w_lambda.to(torch.bfloat16).to(torch.float32)
    b_lambda = torch.zeros(wl.H, device=device)
    c_lambda = torch.full((wl.H,), 0.3, device=device)
    return dict(hidden=hidden, w1=w1.contiguous(), b1=b1.contiguous(),
                w2=w2.contiguous(), b2=b2.contiguous(),
                w_lambda=w_lambda.contiguous(), b_lambda=b_lambda,
                c_lambda=c_lambda, lambda_min=1e-6)
