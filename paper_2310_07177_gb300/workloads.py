"""Seeded synthetic inputs shaped like the paper's serving workloads.

The paper's models (LLaMA-160M / Vicuna-7B, TinyLLaMA-1.1B / Vicuna-33B, T5)
and datasets are not used: random logits with the vocabulary sizes of those
models (32000, 32128) and of a 128k-vocabulary model stand in for them, with a
draft/target relation chosen per workload to give a low, moderate or high
acceptance rate.  This module only draws random numbers (torch generators,
seeded per workload); it computes nothing of the method itself.  Draft tokens
are drawn from softmax(draft / T) with the Gumbel-max trick, i.e. as the draft
model would propose them.

Workloads (seed = 2310071770 + id):

  1 tiny:    verify B=4, k=4, V=32000 fp32, z ~ N(0, 2^2), t = z + N(0, 1), T = 1;
             forward-KL distill of the 16 draft rows against target rows 0..k-1.
  2 verify:  B=32, k=5, V=32000 bf16, z ~ N(0, 2.5^2), t = 0.7 z + N(0, 1.5^2);
             T = 1, plus a greedy (T = 0) pass with the draft argmax as proposals.
  3 flush:   distill N=16384 x V=32128 bf16, z ~ N(0, 2^2), t ~ N(0, 1) with +8 on
             one random entry per row; JSD beta = 0.5; exactly round(0.4 N) rows active.
  4 flush-L: distill N=65536 x V=32000 bf16, z ~ N(0, 2^2), t = z + N(0, 2^2);
             reverse KL and TVD; every row active.
  5 large-V: verify B=256, k=8, V=128256 bf16, z ~ N(0, 3^2), t = 0.5 z + N(0, 2^2),
             T = 0.7; the verify mismatch mask drives forward-KL distill of the
             [B, k] draft rows against target[:, :k].

bf16 rounding is applied to the draft before the target is derived from it.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import torch

SEED_BASE = 2310071770


@dataclass(frozen=True)
class VerifySpec:
    B: int
    k: int
    V: int
    dtype: torch.dtype
    draft_std: float
    target_scale: float  # t = target_scale * z + N(0, target_noise^2)
    target_noise: float
    temperature: float


@dataclass(frozen=True)
class DistillSpec:
    N: int
    V: int
    dtype: torch.dtype
    draft_std: float
    target: str          # "draft+noise" or "peaked"
    target_noise: float
    active_frac: float   # 1.0 = no mask


VERIFY = {
    1: VerifySpec(4, 4, 32000, torch.float32, 2.0, 1.0, 1.0, 1.0),
    2: VerifySpec(32, 5, 32000, torch.bfloat16, 2.5, 0.7, 1.5, 1.0),
    5: VerifySpec(256, 8, 128256, torch.bfloat16, 3.0, 0.5, 2.0, 0.7),
}
DISTILL = {
    3: DistillSpec(16384, 32128, torch.bfloat16, 2.0, "peaked", 1.0, 0.4),
    4: DistillSpec(65536, 32000, torch.bfloat16, 2.0, "draft+noise", 2.0, 1.0),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randn(shape, g, device, chunk_rows: int = 4096):
    """Standard normals in fp32, generated in row chunks to bound peak memory."""
    out = torch.empty(shape, dtype=torch.float32, device=device)
    flat = out.view(-1, shape[-1])
    for r0 in range(0, flat.shape[0], chunk_rows):
        flat[r0:r0 + chunk_rows].normal_(generator=g)
    return out


def verify_inputs(spec: VerifySpec, seed: int, device="cpu", B: Optional[int] = None,
                  V: Optional[int] = None, k: Optional[int] = None) -> dict:
    """draft [B,k,V], target [B,k+1,V], tokens [B,k] int32 (sampled from the
    draft at spec.temperature), greedy_tokens [B,k] (draft argmax),
    uniforms [B,k+1] fp32 in [0,1).  B, V, k override the spec's sizes."""
    B = spec.B if B is None else B
    V = spec.V if V is None else V
    k = spec.k if k is None else k
    g = _gen(seed, device)
    zf = _randn((B, k + 1, V), g, device).mul_(spec.draft_std)
    z = zf.to(spec.dtype)
    # .float() aliases an fp32 tensor, so derive the target out of place
    t = z.float() * spec.target_scale + _randn((B, k + 1, V), g, device).mul_(spec.target_noise)
    t = t.to(spec.dtype)
    draft = z[:, :k].contiguous()
    del zf
    # proposals y_i ~ softmax(z_i / T) by Gumbel-max; greedy proposals = argmax z_i
    T = spec.temperature if spec.temperature > 0 else 1.0
    tokens = torch.empty(B, k, dtype=torch.int32, device=device)
    for i in range(k):
        u = torch.rand(B, V, generator=g, device=device).clamp_(min=1e-12)
        gum = -torch.log(-torch.log(u))
        tokens[:, i] = torch.argmax(draft[:, i].float() / T + gum, dim=-1).to(torch.int32)
    greedy = torch.argmax(draft.float(), dim=-1).to(torch.int32)
    uniforms = torch.rand(B, k + 1, generator=g, device=device, dtype=torch.float32)
    return {"draft": draft, "target": t.contiguous(), "tokens": tokens, "greedy_tokens": greedy,
            "uniforms": uniforms, "temperature": spec.temperature}


def distill_inputs(spec: DistillSpec, seed: int, device="cpu", N: Optional[int] = None,
                   V: Optional[int] = None) -> dict:
    """draft [N,V], target [N,V] and mask [N] uint8 (None when every row is active)."""
    N = spec.N if N is None else N
    V = spec.V if V is None else V
    g = _gen(seed, device)
    z = _randn((N, V), g, device).mul_(spec.draft_std).to(spec.dtype)
    if spec.target == "peaked":
        tf = _randn((N, V), g, device).mul_(spec.target_noise)
        hot = torch.randint(0, V, (N,), generator=g, device=device)
        tf[torch.arange(N, device=device), hot] += 8.0
        t = tf.to(spec.dtype)
        del tf
    else:
        t = (z.float() + _randn((N, V), g, device).mul_(spec.target_noise)).to(spec.dtype)
    mask = None
    if spec.active_frac < 1.0:
        n_on = int(round(spec.active_frac * N))
        perm = torch.randperm(N, generator=g, device=device)
        mask = torch.zeros(N, dtype=torch.uint8, device=device)
        mask[perm[:n_on]] = 1
    return {"draft": z, "target": t, "mask": mask}


def seed_for(config_id: int) -> int:
    return SEED_BASE + config_id


def accepted_inputs(B: int, k: int, seed: int, p_bad: float = 0.05, p_all: float = 0.25) -> torch.Tensor:
    """Accepted counts [B] int32 on the CPU as verification reports them: -1
    (a bad draft token) with probability p_bad, k (every token accepted) with
    probability p_all, otherwise uniform over 0..k-1."""
    g = _gen(seed, "cpu")
    u = torch.rand(B, generator=g)
    a = torch.randint(0, k, (B,), generator=g, dtype=torch.int32)
    a[u < p_all + p_bad] = k
    a[u < p_bad] = -1
    return a


def tree_from_branching(branching) -> list:
    """Parent array of a static candidate tree in breadth-first order.  branching
    is a nested list: branching[d][i] is the number of children of the i-th
    node at depth d (nodes of a depth in order); e.g. [[3], [2, 1, 0]] is a
    root with three candidates, the first with two continuations, the second
    with one."""
    parent = [-1]
    level = [0]
    for counts in branching:
        nxt = []
        for node, c in zip(level, counts):
            for _ in range(c):
                parent.append(node)
                nxt.append(len(parent) - 1)
        level = nxt
    return parent


# A Medusa-style static tree of 26 candidates (27 nodes with the root): 4
# candidates for the next token, 3 / 2 / 1 / 1 continuations of them, and so on
# down to depth 5.
MEDUSA_TREE = tree_from_branching([[4], [3, 2, 1, 1], [2, 1, 1, 1, 1, 0, 1], [2, 1, 1, 0, 1, 0, 1],
                                   [1, 1, 0, 0, 0, 0]])


def tree_inputs(B: int, parent, V: int, dtype, temperature: float, seed: int, device="cpu",
                draft_std: float = 2.0, target_scale: float = 1.0, target_noise: float = 1.0) -> dict:
    """draft [B,n,V], target [B,n,V], tokens [B,n] int32 and uniforms [B,n] for
    the tree `parent`: the children of node i are independent draws from
    softmax(draft row i / T), as a multi-candidate proposer makes them (at
    T = 0 the first child is the draft argmax, the others draws at T = 1)."""
    n = len(parent)
    g = _gen(seed, device)
    z = _randn((B, n, V), g, device).mul_(draft_std)
    t = (z * target_scale + _randn((B, n, V), g, device).mul_(target_noise)).to(dtype)
    z = z.to(dtype)
    T = temperature if temperature > 0 else 1.0
    tokens = torch.zeros(B, n, dtype=torch.int32, device=device)
    for i in range(1, n):
        u = torch.rand(B, V, generator=g, device=device).clamp_(min=1e-12)
        gum = -torch.log(-torch.log(u))
        first = parent.index(parent[i]) == i
        if temperature == 0 and first:
            tokens[:, i] = torch.argmax(z[:, parent[i]].float(), dim=-1).to(torch.int32)
        else:
            tokens[:, i] = torch.argmax(z[:, parent[i]].float() / T + gum, dim=-1).to(torch.int32)
    uniforms = torch.rand(B, n, generator=g, device=device, dtype=torch.float32)
    return {"draft": z.contiguous(), "target": t.contiguous(), "tokens": tokens, "uniforms": uniforms,
            "parent": list(parent), "temperature": temperature}
