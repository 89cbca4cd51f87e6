"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds no arithmetic of the method (no softmax, threshold or
commit logic): it only draws the LM-head weight and per-step hidden states
that both the oracle and the CUDA path consume.  The paper's own inputs are
the final hidden states of LLaDA-8B-Instruct / Dream-7B-Instruct on GSM8K,
HumanEval and LongBench prompts (Section 5); none of those models or datasets
is used here, these generators stand in for them.

Recipe (per workload preset, all seeded):
  * LM-head weight W [V, H]: N(0, 0.02^2), cast to bf16.
  * For every (sequence, block, position) a target token t_p ~ U{0..V-1}
    and a base strength a0_p from the preset's distribution.
  * Hidden state at local step s:
        h = gamma * RMSnorm(kappa * a_p(s) * W[t_p] + n),  n ~ N(0, I_H)
    with a_p(s) = a0_p + 0.5 s (+ a per-block shift for the long preset), the
    noise n fresh for every (sequence, block, position, step), then cast to
    bf16.  kappa = gamma = 1 is the literal recipe; the calibrated recipe uses
    per-shape constants (``CALIBRATED``) that spread first-step confidences
    over all three budget tiers of Box 5 (see ``oracle/calibrate_synth.py``).
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch

SIGMA_W = 0.02


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    V: int
    gen_len: int
    P: int
    T: int
    a0: str               # "u04" | "bimodal" | "long"
    seed_w: int = 1234
    seed_h: int = 0

    @property
    def n_blocks(self) -> int:
        return self.gen_len // self.P


# Shapes of the five configurations of the spec workload list.
WORKLOADS = {
    "toy": Workload("toy", B=1, H=256, V=4096, gen_len=64, P=16, T=8, a0="u04"),
    "llada": Workload("llada", B=1, H=4096, V=126464, gen_len=256, P=32, T=32, a0="u04"),
    "dream": Workload("dream", B=1, H=3584, V=152064, gen_len=256, P=32, T=32, a0="bimodal"),
    "llada_batched": Workload("llada_batched", B=64, H=4096, V=126464, gen_len=256, P=32, T=32,
                              a0="u04"),
    "dream_long": Workload("dream_long", B=8, H=3584, V=152064, gen_len=1024, P=64, T=64,
                           a0="long"),
}

# (kappa, gamma) per (V, H), written by oracle/calibrate_synth.py.
CALIBRATED: dict[tuple[int, int], tuple[float, float]] = {
    (4096, 256): (12.494524, 3.125000),
    (126464, 4096): (3.612477, 0.781250),
    (152064, 3584): (3.891420, 0.835191),
}


def gains(V: int, H: int, mode: str) -> tuple[float, float]:
    if mode == "literal":
        return 1.0, 1.0
    if mode == "calibrated":
        if (V, H) in CALIBRATED:
            return CALIBRATED[(V, H)]
        return default_gains(V, H)
    raise ValueError(mode)


def default_gains(V: int, H: int) -> tuple[float, float]:
    """Gains from the first-order closed form, used for shapes with no stored
    calibration: gamma sets the off-target logit spread to 1, kappa puts the
    median first-step confidence of a token with a = 2.75 near 1/2."""
    s0 = SIGMA_W * math.sqrt(H)
    gamma = 1.0 / s0
    lse_bg = math.log(V) + 0.5
    beta = lse_bg / 2.75               # logit lift per unit strength
    kappa = beta / (gamma * SIGMA_W * SIGMA_W * H)
    return kappa, gamma


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & ((1 << 63) - 1))
    return g


def lm_head_weight(V: int, H: int, seed: int = 1234, device="cpu", chunk_rows: int = 8192):
    """W [V, H] bf16 with entries N(0, 0.02^2), generated in row chunks."""
    W = torch.empty((V, H), dtype=torch.bfloat16, device=device)
    g = _gen(seed, device)
    for r in range(0, V, chunk_rows):
        n = min(chunk_rows, V - r)
        W[r:r + n] = (torch.randn((n, H), generator=g, device=device, dtype=torch.float32)
                      * SIGMA_W).to(torch.bfloat16)
    return W


def _a0(kind: str, shape, g, device):
    u = torch.rand(shape, generator=g, device=device, dtype=torch.float64)
    if kind in ("u04", "long"):
        return 4.0 * u
    if kind == "bimodal":
        pick = torch.rand(shape, generator=g, device=device, dtype=torch.float64)
        hi = 3.0 + 3.0 * u
        lo = 1.5 * u
        return torch.where(pick < 0.6, hi, lo)
    raise ValueError(kind)


class HiddenStates:
    """Per-step hidden states [B, P, H] bf16 for a workload."""

    def __init__(self, wl: Workload, W: torch.Tensor, mode: str = "calibrated", seed: int | None = None):
        self.wl = wl
        self.W = W
        self.device = W.device
        self.kappa, self.gamma = gains(wl.V, wl.H, mode)
        self.seed = wl.seed_h if seed is None else seed
        g = _gen(self.seed * 1000003 + 17, self.device)
        shape = (wl.B, wl.n_blocks, wl.P)
        self.targets = torch.randint(0, wl.V, shape, generator=g, device=self.device, dtype=torch.int64)
        self.a0 = _a0(wl.a0, shape, g, self.device)
        if wl.a0 == "long":
            # Later blocks are easier: the base strength rises by 0.25 per block.
            self.a0 = self.a0 + 0.25 * torch.arange(wl.n_blocks, device=self.device,
                                                    dtype=torch.float64)[None, :, None]

    def strength(self, blk: int, s: int) -> torch.Tensor:
        return self.a0[:, blk, :] + 0.5 * s

    def __call__(self, blk: int, s: int, out: torch.Tensor | None = None) -> torch.Tensor:
        wl = self.wl
        g = _gen((self.seed * 7919 + blk) * 104729 + s, self.device)
        n = torch.randn((wl.B, wl.P, wl.H), generator=g, device=self.device, dtype=torch.float32)
        a = self.strength(blk, s).to(torch.float32)
        tgt = self.W[self.targets[:, blk, :].reshape(-1)].to(torch.float32).reshape(wl.B, wl.P, wl.H)
        x = self.kappa * a[..., None] * tgt + n
        x = x * torch.rsqrt(torch.mean(x * x, dim=-1, keepdim=True))
        h = (self.gamma * x).to(torch.bfloat16)
        if out is not None:
            out.copy_(h)
            return out
        return h


# ---------------------------------------------------------------- final norm --

def final_norm_weight(H: int, seed: int = 5, device="cpu") -> torch.Tensor:
    """Stand-in for the weight of a model's final RMSNorm: 1 + 0.15 N(0, 1), bf16."""
    g = _gen(seed * 7 + 3, device)
    return (1.0 + 0.15 * torch.randn(H, generator=g, device=device,
                                     dtype=torch.float32)).to(torch.bfloat16)


class PreNormHidden:
    """The rows of a ``HiddenStates`` generator times a fixed positive scale per
    position (0.3 to 3.0): a stand-in for the last layer's output before the
    model's final RMSNorm, which removes the scale again."""

    def __init__(self, hs: HiddenStates, seed: int = 21):
        wl = hs.wl
        g = _gen(seed * 13 + 5, hs.device)
        self.hs = hs
        self.wl = wl
        self.scale = 0.3 + 2.7 * torch.rand((wl.B, wl.P, 1), generator=g, device=hs.device,
                                            dtype=torch.float32)

    def __call__(self, blk: int, s: int) -> torch.Tensor:
        return (self.hs(blk, s).to(torch.float32) * self.scale).to(torch.bfloat16)
