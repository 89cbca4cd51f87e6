"""Run the first steps of a workload's first block through the C ABI, for
profiler captures of single kernels with a bounded device footprint.

    python -m paper_2608_22646_gb300.profile_step --workload llada_batched --steps 3

The weight is generated once; each step's hidden states are generated just
before its step call (unlike ``bench.py``, which holds a whole generation's
inputs on the device and times it).  Prints the masked-row count M_t of every
step that ran, so a captured launch can be matched to its size.  Times nothing.
"""
from __future__ import annotations

import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main(argv=None) -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="llada_batched")
    ap.add_argument("--steps", type=int, default=3)
    args = ap.parse_args(argv)
    import torch
    import synth
    import paper_2608_22646_gb300 as cai

    wl = synth.WORKLOADS[args.workload]
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device="cuda")
    hs = synth.HiddenStates(wl, W, "calibrated")
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    ctx = cai.cai_init(cfg, W)
    try:
        ran = 0
        for t in range(min(args.steps, wl.T)):
            h = hs(0, t)
            torch.cuda.synchronize()
            if t == 0:
                cai.cai_first_step(ctx, h)
            else:
                cai.cai_denoise_step(ctx, h)
            ran += 1
            if cai.cai_poll(ctx, 0, 60000):
                break
        st = cai.cai_state_download(ctx)
        print(json.dumps({"workload": wl.name, "steps": ran,
                          "M": [int(m) for m in st["m_hist"][0, :ran]],
                          "stats": cai.cai_get_stats(ctx)}))
    finally:
        cai.cai_free(ctx)
    return 0


if __name__ == "__main__":
    sys.exit(main())
