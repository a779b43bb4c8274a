"""Seeded synthetic logits shaped like the paper's serving workloads.

This module only draws inputs; it holds none of the feedback or learner
arithmetic, and both the CUDA path's tests/benchmark and the oracle's tests
take their inputs from it.  No dataset or trained weight is used: the
paper's drafters are domain-finetuned EAGLE-3 heads that are accurate in
their own domain and poor elsewhere (Sec. 4.1), which the recipes imitate
with a drafter = target + Gaussian noise whose scale depends on whether the
query's domain is the drafter's.

Recipes (all logits drawn in fp32, then rounded to the storage dtype):
  * target, "gauss":  z ~ N(0, 3^2) i.i.d.
  * target, "zipf":   z_v = -1.1 ln(rank_v) + N(0, 2^2), rank a per-row random
                      permutation of 1..V (a heavy-tailed LM-like row whose
                      argmax position differs from row to row)
  * drafter i, query b:  z_target + N(0, sigma[i,b]^2) at every position.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

DTYPES = {"bf16": torch.bfloat16, "fp16": torch.float16, "fp32": torch.float32}


@dataclass(frozen=True)
class Workload:
    name: str
    N: int
    B: int
    P: int                      # K + 1 verified positions
    V: int
    dtype: str
    temperature: float
    target: str                 # "gauss" | "zipf"
    sigma: str                  # how sigma[i,b] is set, see drafter_sigma()
    greedy: tuple = (False,)    # feedback modes the workload runs
    learner: str = "normalhedge"
    eta: float = 0.0
    rounds: int = 1
    M: int = 0                  # tree nodes per query (0 = chain)
    seed_base: int = 0
    note: str = field(default="", compare=False)

    @property
    def K(self) -> int:
        return self.P - 1

    @property
    def rows(self) -> int:
        return self.B * self.P * (self.N + 1)

    @property
    def evals(self) -> int:
        """drafter-position-vocab evaluations per feedback call, N*B*P*V"""
        return self.N * self.B * self.P * self.V

    @property
    def bytes_per_call(self) -> int:
        """every target and drafter logit read once"""
        return self.rows * self.V * (4 if self.dtype == "fp32" else 2)


WORKLOADS = {
    "tiny_chain": Workload(
        "tiny_chain", N=2, B=1, P=5, V=1000, dtype="fp32", temperature=1.0, target="gauss",
        sigma="tiny", greedy=(False, True), learner="hedge", eta=0.5, rounds=50, seed_base=0,
        note="N=2 B=1 K=4 V=1000 fp32, sigma=(0.5,2.0), T=1 and greedy, Hedge eta=0.5, 50 rounds"),
    "qwen3_8b_chain": Workload(
        "qwen3_8b_chain", N=4, B=8, P=7, V=151936, dtype="bf16", temperature=0.7, target="zipf",
        sigma="qwen", seed_base=2000,
        note="N=4 B=8 K=6 V=151936 bf16, sigma in {0.3,1,2,4}, T=0.7"),
    "llama3_batch": Workload(
        "llama3_batch", N=8, B=64, P=9, V=128256, dtype="bf16", temperature=1.0, target="zipf",
        sigma="domain", greedy=(False, True), learner="normalhedge", seed_base=3000,
        note="N=8 B=64 K=8 V=128256 bf16, domain b mod 8 (sigma 0.3 vs 2.5), T=1 and greedy"),
    "tree_path": Workload(
        "tree_path", N=16, B=32, P=4, V=151936, dtype="bf16", temperature=1.0, target="zipf",
        sigma="uniform", M=85, seed_base=4000,
        note="N=16 B=32, 4-4-4 tree (85 nodes, 64 leaves), path of 4, V=151936 bf16"),
    "long_session": Workload(
        "long_session", N=8, B=128, P=6, V=151936, dtype="bf16", temperature=1.0, target="zipf",
        sigma="switching", learner="both", eta=math.sqrt(8 * math.log(8) / 2000), rounds=2000,
        seed_base=5000,
        note="N=8 B=128 K=5 V=151936 bf16, 2000 rounds, expert (b + t//250) mod 8"),
}


def drafter_sigma(w: Workload, gen: torch.Generator, rnd: int = 0, B: int | None = None,
                  N: int | None = None) -> torch.Tensor:
    """sigma[i,b] (CPU fp32) for round rnd."""
    N = w.N if N is None else N
    B = w.B if B is None else B
    i = torch.arange(N)[:, None]
    b = torch.arange(B)[None, :]
    if w.sigma == "tiny":
        base = torch.tensor([0.5, 2.0] + [2.0] * max(0, N - 2))[:N]
        return base[:, None].expand(N, B).clone()
    if w.sigma == "qwen":
        base = torch.tensor([0.3, 1.0, 2.0, 4.0] * ((N + 3) // 4))[:N]
        return base[:, None].expand(N, B).clone()
    if w.sigma == "domain":
        return torch.where(i == (b % N), 0.3, 2.5).float()
    if w.sigma == "switching":
        return torch.where(i == ((b + rnd // 250) % N), 0.3, 2.5).float()
    if w.sigma == "uniform":
        s = 0.2 + 2.8 * torch.rand(N, generator=gen)
        return s[:, None].expand(N, B).clone()
    raise ValueError(w.sigma)


def _target_rows(kind: str, rows: int, V: int, gen: torch.Generator, device) -> torch.Tensor:
    if kind == "gauss":
        return 3.0 * torch.randn(rows, V, generator=gen, device=device)
    rank_of = torch.rand(rows, V, generator=gen, device=device).argsort(dim=1)
    offset = -1.1 * torch.log(torch.arange(1, V + 1, device=device, dtype=torch.float32))
    z = torch.empty(rows, V, device=device, dtype=torch.float32)
    z.scatter_(1, rank_of, offset.expand(rows, V))
    return z.add_(2.0 * torch.randn(rows, V, generator=gen, device=device))


def tree_path_indices(B: int, gen: torch.Generator, branching=(4, 4, 4)) -> torch.Tensor:
    """[B, depth+1] int32 node ids of a random root-to-leaf path; nodes are
    numbered level by level (root 0, then its children, ...)."""
    depth = len(branching)
    out = torch.zeros(B, depth + 1, dtype=torch.int32)
    for b in range(B):
        first, node_in_level = 0, 0
        level_size = 1
        for d, L in enumerate(branching):
            first += level_size
            node_in_level = node_in_level * L + int(torch.randint(L, (1,), generator=gen))
            level_size *= L
            out[b, d + 1] = first + node_in_level
    return out


def make_inputs(w: Workload, rnd: int = 0, device="cpu", seed: int | None = None,
                B: int | None = None, N: int | None = None, P: int | None = None,
                V: int | None = None, sigma: torch.Tensor | None = None) -> dict:
    """One round of logits.  Returns a dict with 'target' ([B,P,V], or the
    tree [B,M,V] with 'path' [B,P] int32), 'drafter' [N,B,P,V] in the
    workload's dtype on `device`, and 'sigma' [N,B].  Sizes may be overridden
    for reduced test cases; the seed defaults to seed_base + rnd."""
    N = w.N if N is None else N
    B = w.B if B is None else B
    P = w.P if P is None else P
    V = w.V if V is None else V
    seed = w.seed_base + rnd if seed is None else seed
    dt = DTYPES[w.dtype]
    cpu_gen = torch.Generator().manual_seed(seed)
    gen = torch.Generator(device=device).manual_seed(seed + 7919)
    if sigma is None:
        sigma = drafter_sigma(w, cpu_gen, rnd, B=B, N=N)
    out = {"sigma": sigma}
    if w.M:
        M = w.M
        tree = _target_rows(w.target, B * M, V, gen, device).view(B, M, V)
        path = tree_path_indices(B, cpu_gen)
        assert path.shape[1] == P, "tree depth + 1 must equal P"
        out["path"] = path.to(device)
        tgt32 = torch.stack([tree[b, path[b].long().to(device)] for b in range(B)])
        out["target"] = tree.to(dt)
        del tree
    else:
        tgt32 = _target_rows(w.target, B * P, V, gen, device).view(B, P, V)
        out["target"] = tgt32.to(dt)
    drafter = torch.empty((N, B, P, V), device=device, dtype=dt)
    sig = sigma.to(device)
    for i in range(N):
        noise = torch.randn(B, P, V, generator=gen, device=device)
        drafter[i] = (tgt32 + sig[i][:, None, None] * noise).to(dt)
    out["drafter"] = drafter
    return out


def storage_numpy(t: torch.Tensor):
    """Stored bytes of a logit tensor as numpy (bf16 -> uint16 bit patterns)."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view("uint16")
    return t.numpy()
