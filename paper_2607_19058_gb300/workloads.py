"""Seeded synthetic workloads shaped like the paper's MoE parameter sets.

This module only describes tensors (shapes, tiers) and draws seeded inputs
(weights, gradients); it holds none of the optimizer's arithmetic, so both the
CUDA path and the CPU oracle can be fed from it.

Shape sets:
  * ``toy``      -- a tiny MoE (embedding 512x64, experts 8 x {64x128, 64x128, 128x64},
                    router 64x8), for exhaustive parity;
  * ``slice``    -- one MoE layer of the full model (128 experts x {4096x1024,
                    1024x4096, 4096x1024}, one attention block, router 4096x128);
  * ``appb``     -- the paper's 6.78B model by tier (App. B parameter counts: embedding
                    50304x4096 tied, positions 256x4096, 2 x GQA attention, dense SwiGLU
                    FFN, 10 norm vectors, 128 x 3 experts of 4096x4096, router 4096x128);
  * ``literal``  -- the shape list as a literal reading of "32 attention/FFN matrices of
                    4096x4096 plus a 32000x4096 embedding" (7.11B parameters);
  * ``skewed``   -- ``appb`` shapes with Zipf-skewed expert loads (zero-grad experts,
                    heavy-tailed grads, periodic 100x router spikes);
  * ``ablation`` -- ``appb`` with expert momentum and awkward shapes (embedding
                    50257x4096, 4095x1000, 1x4096, router 4096x127).

The paper trains on OpenWebText; its gradients are not available, so these seeded
distributions stand in for them with the paper's exact parameter shapes.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import torch

TIER_BACKBONE, TIER_EXPERT, TIER_ROUTER = 0, 1, 2
POLICY_TIERED, POLICY_EXPERT_MOMENTUM, POLICY_FACTORED_ROUTER, POLICY_UNIFORM, POLICY_ADAFACTOR = 0, 1, 2, 3, 4


@dataclasses.dataclass(frozen=True)
class Spec:
    name: str
    shape: Tuple[int, ...]
    tier: int
    expert: int = -1          # expert index for expert tensors
    no_decay: bool = False
    fp32: bool = False        # weights and gradient kept in fp32 (App. A: norms and router)

    @property
    def dtype(self):
        return torch.float32 if self.fp32 else torch.bfloat16

    @property
    def numel(self) -> int:
        return math.prod(self.shape)


@dataclasses.dataclass(frozen=True)
class HP:
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-30
    clip_d: float = 1.0
    weight_decay: float = 0.1
    lr: float = 1e-3
    policy: int = POLICY_TIERED


@dataclasses.dataclass
class Workload:
    name: str
    specs: List[Spec]
    hp: HP
    grad_kind: str            # "normal", "toy", "slice", "skewed"
    steps: int
    seed: int = 0
    n_experts: int = 0

    @property
    def numel(self) -> int:
        return sum(s.numel for s in self.specs)


# --------------------------------------------------------------------------
# Shape sets
# --------------------------------------------------------------------------
def _attention(prefix, d, kv):
    return [Spec(f"{prefix}.q", (d, d), TIER_BACKBONE), Spec(f"{prefix}.k", (kv, d), TIER_BACKBONE),
            Spec(f"{prefix}.v", (kv, d), TIER_BACKBONE), Spec(f"{prefix}.o", (d, d), TIER_BACKBONE)]


def _norm(prefix, d):
    return [Spec(f"{prefix}.weight", (d,), TIER_BACKBONE), Spec(f"{prefix}.bias", (d,), TIER_BACKBONE)]


def _experts(n_exp, shapes):
    out = []
    for e in range(n_exp):
        for k, shp in enumerate(shapes):
            out.append(Spec(f"expert{e}.w{k}", tuple(shp), TIER_EXPERT, expert=e))
    return out


def toy() -> Workload:
    d = 64
    specs = [Spec("embed", (512, d), TIER_BACKBONE),
             Spec("attn.qkv", (d, 192), TIER_BACKBONE), Spec("attn.o", (d, d), TIER_BACKBONE),
             Spec("ffn.up", (d, 256), TIER_BACKBONE), Spec("ffn.down", (256, d), TIER_BACKBONE),
             Spec("norm.attn", (d,), TIER_BACKBONE), Spec("norm.ffn", (d,), TIER_BACKBONE),
             Spec("norm.final", (d,), TIER_BACKBONE),
             Spec("router", (d, 8), TIER_ROUTER)]
    specs += _experts(8, [(d, 128), (d, 128), (128, d)])
    return Workload("toy", specs, HP(), "toy", steps=10, n_experts=8)


def slice_() -> Workload:
    d = 4096
    specs = _attention("attn", d, d) + [Spec("norm.attn", (d,), TIER_BACKBONE),
                                        Spec("norm.ffn", (d,), TIER_BACKBONE),
                                        Spec("router", (d, 128), TIER_ROUTER)]
    specs += _experts(128, [(d, 1024), (1024, d), (d, 1024)])
    return Workload("slice", specs, HP(), "slice", steps=20, n_experts=128)


def _appb_specs(vocab=50304, router_cols=128, extra=()):
    d, kv = 4096, 1024
    specs = [Spec("embed", (vocab, d), TIER_BACKBONE), Spec("pos", (256, d), TIER_BACKBONE)]
    # block 0: attention + dense SwiGLU FFN
    specs += _norm("b0.ln1", d) + _attention("b0.attn", d, kv) + _norm("b0.ln2", d)
    specs += [Spec("b0.ffn.gate", (d, d), TIER_BACKBONE), Spec("b0.ffn.up", (d, d), TIER_BACKBONE),
              Spec("b0.ffn.down", (d, d), TIER_BACKBONE)]
    # block 1: attention + MoE
    specs += _norm("b1.ln1", d) + _attention("b1.attn", d, kv) + _norm("b1.ln2", d)
    specs += [Spec("b1.router", (d, router_cols), TIER_ROUTER)]
    specs += _experts(128, [(d, d), (d, d), (d, d)])
    specs += _norm("ln_f", d)
    specs += list(extra)
    return specs


def appb() -> Workload:
    return Workload("appb", _appb_specs(), HP(), "normal", steps=50, n_experts=128)


def literal() -> Workload:
    d = 4096
    specs = [Spec("embed", (32000, d), TIER_BACKBONE)]
    specs += [Spec(f"mat{k}", (d, d), TIER_BACKBONE) for k in range(32)]
    specs += [Spec(f"norm{k}", (d,), TIER_BACKBONE) for k in range(10)]
    specs += [Spec("router", (d, 128), TIER_ROUTER)]
    specs += _experts(128, [(d, d), (d, d), (d, d)])
    return Workload("literal", specs, HP(), "normal", steps=50, n_experts=128)


def skewed() -> Workload:
    return Workload("skewed", _appb_specs(), HP(), "skewed", steps=50, n_experts=128)


def ablation() -> Workload:
    extra = [Spec("odd.a", (4095, 1000), TIER_BACKBONE), Spec("odd.b", (1, 4096), TIER_BACKBONE)]
    specs = _appb_specs(vocab=50257, router_cols=127, extra=extra)
    return Workload("ablation", specs, HP(policy=POLICY_EXPERT_MOMENTUM), "normal", steps=20, n_experts=128)


def toy_fp32() -> Workload:
    """The toy set with the router and the norm vectors kept in fp32 (App. A)."""
    wl = toy()
    specs = [dataclasses.replace(s, fp32=True) if (s.tier == TIER_ROUTER or len(s.shape) == 1) else s
             for s in wl.specs]
    return dataclasses.replace(wl, name="toy_fp32", specs=specs)


def appb_fp32() -> Workload:
    """The App. B shapes at the paper's precision: router and LayerNorm vectors fp32 (App. A)."""
    wl = appb()
    specs = [dataclasses.replace(s, fp32=True) if (s.tier == TIER_ROUTER or len(s.shape) == 1) else s
             for s in wl.specs]
    return dataclasses.replace(wl, name="appb_fp32", specs=specs)


def adafactor() -> Workload:
    """The App. B shapes under the Adafactor comparator (Sec. 5, App. A): every matrix
    factored, no momentum, beta2_t = 1 - t^-0.8."""
    return Workload("adafactor", _appb_specs(), HP(policy=POLICY_ADAFACTOR), "normal", steps=20, n_experts=128)


def small() -> Workload:
    """A 558M-parameter cut of the App. B set (32 experts, a 4096^2 and a 1024x4096 backbone
    matrix, 2 norm vectors, the router): 2.2 GB of weights + gradients, well above L2,
    for profiler captures that must stay small."""
    d = 4096
    specs = [Spec("b.q", (d, d), TIER_BACKBONE), Spec("b.k", (1024, d), TIER_BACKBONE)] + _norm("ln", d)
    specs += [Spec("router", (d, 128), TIER_ROUTER)]
    specs += _experts(32, [(d, d)])
    return Workload("small", specs, HP(), "normal", steps=20, n_experts=32)


def stack_experts(wl: Workload) -> Workload:
    """The same parameter set with each expert weight kept as one (E, n, m) array
    over the experts (how MoE layers usually store them); other tensors as they are."""
    shapes, rest, first = {}, [], None
    for k, s in enumerate(wl.specs):
        if s.tier == TIER_EXPERT and s.expert >= 0:
            slot = s.name.rsplit(".", 1)[1]
            shapes.setdefault(slot, (s.shape, []))[1].append(s.expert)
            first = len(rest) if first is None else first
        else:
            rest.append(s)
    stacks = [Spec(f"experts.{slot}", (len(es),) + tuple(shp), TIER_EXPERT) for slot, (shp, es) in shapes.items()]
    specs = rest[:first] + stacks + rest[first:] if stacks else rest
    return dataclasses.replace(wl, name=wl.name + "_stacked", specs=specs, grad_kind="normal")


WORKLOADS = {"small": small, "toy": toy, "slice": slice_, "appb": appb, "literal": literal, "skewed": skewed,
             "ablation": ablation, "adafactor": adafactor, "toy_fp32": toy_fp32, "appb_fp32": appb_fp32}


def get(name: str) -> Workload:
    return WORKLOADS[name]()


# --------------------------------------------------------------------------
# Seeded draws
# --------------------------------------------------------------------------
def _mix(*xs: int) -> int:
    """Deterministic 63-bit seed from integers (splitmix-style)."""
    h = 0x9E3779B97F4A7C15
    for x in xs:
        h ^= (x + 0x632BE59BD9B4E019 + (h << 6) + (h >> 2)) & 0xFFFFFFFFFFFFFFFF
        h = (h * 0xBF58476D1CE4E5B9) & 0xFFFFFFFFFFFFFFFF
        h ^= h >> 31
    return h & 0x7FFFFFFFFFFFFFFF


def _gen(device, *xs) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_mix(*xs))
    return g


def _normal(shape, std, gen, device) -> torch.Tensor:
    return (torch.randn(shape, generator=gen, device=device, dtype=torch.float32) * std)


def init_weight(wl: Workload, tid: int, device="cpu") -> torch.Tensor:
    """W ~ N(0, 0.02^2), bf16 (fp32 for an fp32 tensor)."""
    s = wl.specs[tid]
    return _normal(s.shape, 0.02, _gen(device, wl.seed, 1, tid), device).to(s.dtype)


def dirichlet_loads(n: int, seed: int) -> torch.Tensor:
    """Expert loads ~ Dirichlet(1) (normalised Exp(1) draws), drawn once, on the CPU."""
    g = _gen("cpu", seed, 7)
    u = torch.rand(n, generator=g, dtype=torch.float64).clamp_min(1e-300)
    e = -torch.log(u)
    return e / e.sum()


def zipf_ranks(n: int, seed: int, step: int) -> torch.Tensor:
    """Per-step seeded permutation: rank (1-based) of each expert under Zipf loads."""
    g = _gen("cpu", seed, 11, step)
    perm = torch.randperm(n, generator=g)
    ranks = torch.empty(n, dtype=torch.int64)
    ranks[perm] = torch.arange(1, n + 1)
    return ranks


def _student_t3(shape, gen, device) -> torch.Tensor:
    z = torch.randn((4,) + tuple(shape), generator=gen, device=device, dtype=torch.float32)
    chi2 = z[1] * z[1] + z[2] * z[2] + z[3] * z[3]
    return z[0] / torch.sqrt(chi2 / 3.0)


def grad(wl: Workload, tid: int, step: int, device="cpu") -> torch.Tensor:
    """Gradient of tensor `tid` at (1-based) `step` per the workload's recipe, bf16 (fp32
    for an fp32 tensor: the same fp32 draw, not rounded)."""
    return _grad32(wl, tid, step, device).to(wl.specs[tid].dtype)


def _grad32(wl: Workload, tid: int, step: int, device) -> torch.Tensor:
    s = wl.specs[tid]
    gen = _gen(device, wl.seed, 2, step, tid)
    if wl.grad_kind == "toy":
        if s.tier == TIER_EXPERT and s.expert in (5, 6, 7) and step % 2 == 1:
            return torch.zeros(s.shape, dtype=torch.float32, device=device)
        return _normal(s.shape, 1e-3, gen, device)
    if wl.grad_kind == "slice":
        if s.tier == TIER_EXPERT:
            load = float(dirichlet_loads(wl.n_experts, wl.seed)[s.expert])
            return _normal(s.shape, 1e-3 * math.sqrt(64.0 * load), gen, device)
        return _normal(s.shape, 1e-3, gen, device)
    if wl.grad_kind == "skewed":
        if s.tier == TIER_EXPERT:
            rank = int(zipf_ranks(wl.n_experts, wl.seed, step)[s.expert])
            if rank > wl.n_experts - 40:      # the 40 least-loaded experts see no tokens
                return torch.zeros(s.shape, dtype=torch.float32, device=device)
            return (1e-3 * _student_t3(s.shape, gen, device))
        g = _normal(s.shape, 1e-3, gen, device)
        if s.tier == TIER_ROUTER and step % 10 == 7:
            g = g * 100.0
        return g
    return _normal(s.shape, 1e-3, gen, device)


def bf16_bits(t: torch.Tensor):
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view("uint16").reshape(-1)
