"""Calibrate the synthetic hidden-state gains (kappa, gamma) on the oracle.

TEST INFRASTRUCTURE ONLY (calls ``oracle`` and ``synth``, nothing else).

The literal generator h = RMSnorm(a W[t] + n) gives every token a first-step
confidence near 1/V (the target's logit lift is tiny against the log-sum-exp
of the V - 1 off-target logits), so every budget is 64 and every block stops at
t = 3 in the grinding detector.  The calibrated generator
h = gamma RMSnorm(kappa a W[t] + n) fixes:

  * gamma = 1 / (0.02 sqrt(H)): off-target logits get unit standard deviation;
  * kappa by bisection (seeded, 40 halvings in log space) so that the median
    oracle confidence of tokens with strength a = 2.75 equals 1/2.

With a0 ~ U(0, 4) this puts first-step confidences in all three tiers of
Box 5 (c < 0.25, 0.25..0.50, > 0.50).  Run as
``python -m oracle.calibrate_synth`` and paste the printed table into
``synth.CALIBRATED``.
"""
from __future__ import annotations

import math
import sys

import numpy as np
import torch

import oracle
import synth

A_MID = 2.75
N_SAMPLES = 48


def median_conf(W: torch.Tensor, kappa: float, gamma: float, seed: int = 99) -> float:
    V, H = W.shape
    g = torch.Generator().manual_seed(seed)
    tgt = torch.randint(0, V, (N_SAMPLES,), generator=g)
    n = torch.randn((N_SAMPLES, H), generator=g, dtype=torch.float32)
    x = kappa * A_MID * W[tgt].to(torch.float32) + n
    x = x * torch.rsqrt(torch.mean(x * x, dim=-1, keepdim=True))
    h = (gamma * x).to(torch.bfloat16)
    return float(np.median(oracle.head_rows(W, h)["conf"]))


def calibrate(V: int, H: int, seed_w: int = 1234, iters: int = 40) -> tuple[float, float]:
    W = synth.lm_head_weight(V, H, seed=seed_w)
    gamma = 1.0 / (synth.SIGMA_W * math.sqrt(H))
    lo, hi = math.log(0.1), math.log(1000.0)
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if median_conf(W, math.exp(mid), gamma) < 0.5:
            lo = mid
        else:
            hi = mid
    return math.exp(0.5 * (lo + hi)), gamma


if __name__ == "__main__":
    names = sys.argv[1:] or ["toy", "llada", "dream"]
    seen = set()
    for name in names:
        wl = synth.WORKLOADS[name]
        if (wl.V, wl.H) in seen:
            continue
        seen.add((wl.V, wl.H))
        k, gm = calibrate(wl.V, wl.H, wl.seed_w)
        print(f"    ({wl.V}, {wl.H}): ({k:.6f}, {gm:.6f}),", flush=True)
