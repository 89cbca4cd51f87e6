"""The allocation-free decoding head, cai_head_rows_static.

It is for callers that cannot call cudaMalloc where they need the head: a
memory pool that already owns the whole device, a runtime that reserved all
memory up front, or a region where an allocation would synchronise the
device.  It allocates nothing, keeping its only scratch in a fixed device
array.  These tests call it through the C ABI and compare its confidences and
argmaxes with the context path (cai_first_step) on the same rows, within the
parity tolerances, on two calls in a row with different inputs.

This file is collected last on purpose; it passes alone in a fresh process
and after the other tests.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2608_22646_gb300 as cai
from tests import parity

pytestmark = pytest.mark.gpu


def _context_head(W, h, P, H, V):
    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, 1, P, H, V, 4, 1)
    ctx = cai.cai_init(cfg, W)
    try:
        cai.cai_first_step(ctx, h)
        torch.cuda.synchronize()
        st = cai.cai_state_download(ctx)
    finally:
        cai.cai_free(ctx)
    return st["s0"][0, :P].copy(), st["cand"][0, :P].copy()


@pytest.mark.parametrize("V,H,P", [(4096, 256, 16), (1000, 128, 33), (2112, 192, 256)])
def test_static_head_matches_context_path_on_two_calls(V, H, P):
    cai.cai_test_head_grid_limit(0)
    W = synth.lm_head_weight(V, H, seed=1234, device="cuda")
    wl = synth.Workload("rows", B=1, H=H, V=V, gen_len=P, P=P, T=4, a0="u04")
    hs = synth.HiddenStates(wl, W, "calibrated", seed=21)
    for t in (0, 2):                                  # two calls, different rows
        h = hs(0, t).reshape(P, H).contiguous()
        ref_conf, ref_arg = _context_head(W, h, P, H, V)
        conf = torch.full((P,), -1.0, dtype=torch.float32, device="cuda")
        arg = torch.full((P,), -7, dtype=torch.int32, device="cuda")
        cai.cai_head_rows_static(W, h, conf, arg)
        torch.cuda.synchronize()
        got_conf, got_arg = conf.cpu().numpy(), arg.cpu().numpy()
        np.testing.assert_allclose(got_conf, ref_conf, rtol=0, atol=parity.CONF_TOL)
        gap = oracle.head_rows(W, h)["gap"]
        sure = gap > parity.GAP_TOL                   # argmax unique beyond 1e-2
        assert np.array_equal(got_arg[sure], ref_arg[sure])


def test_static_head_limits_and_no_allocation():
    V, H, M = 4096, 256, 8
    W = synth.lm_head_weight(V, H, device="cuda")
    rows = (torch.randn((300, H), device="cuda") * 0.5).to(torch.bfloat16)
    conf = torch.empty((300,), dtype=torch.float32, device="cuda")
    arg = torch.empty((300,), dtype=torch.int32, device="cuda")
    with pytest.raises(cai.CaiError) as e:            # more rows than the scratch holds
        cai.cai_head_rows_static(W, rows[:257], conf, arg)
    assert e.value.status == cai.CAI_ERR_SHAPE
    with pytest.raises(cai.CaiError) as e:            # vocabulary below one 128-row tile
        cai.cai_head_rows_static(W[:100], rows[:M], conf, arg)
    assert e.value.status == cai.CAI_ERR_SHAPE
    # The library's allocator is armed to fail its next allocation; the entry
    # point does not use it, so the call still succeeds.
    cai.cai_test_fail_alloc_after(1)
    try:
        cai.cai_head_rows_static(W, rows[:M], conf, arg)
        torch.cuda.synchronize()
    finally:
        cai.cai_test_fail_alloc_after(0)
    o = oracle.head_rows(W, rows[:M])
    assert np.all(np.abs(conf[:M].cpu().numpy() - o["conf"]) <= parity.CONF_TOL)
