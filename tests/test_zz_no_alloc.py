"""The allocation-free decoding head, cai_head_rows_static.

It is for callers that cannot call cudaMalloc where they need the head: a
memory pool that already owns the whole device, a runtime that reserved all
memory up front, or a region where an allocation would synchronise the
device.  It allocates nothing, keeping its only scratch in a fixed device
array.  These tests call it through the C ABI and compare its confidences and
argmaxes, element by element, with the fp64 oracle (conf within 2e-3, argmax
wherever the oracle's top-2 gap exceeds 1e-2) and with the context path
(cai_first_step) on the same rows, on two calls in a row with different
inputs; at full LLaDA / Dream size (several 128-row tiles per CTA, so the
stage ring wraps and both accumulators alternate) the oracle recomputes a
sample of the rows.

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


def _static(W, h):
    M = h.shape[0]
    conf = torch.full((M,), -1.0, dtype=torch.float32, device="cuda")
    arg = torch.full((M,), -7, dtype=torch.int32, device="cuda")
    cai.cai_head_rows_static(W, h, conf, arg)
    torch.cuda.synchronize()
    return conf.cpu().numpy(), arg.cpu().numpy()


def _check_against_oracle(W, h, conf, arg, sample=None):
    rows = h if sample is None else h[sample]
    o = oracle.head_rows(W, rows)
    c, a = (conf, arg) if sample is None else (conf[sample], arg[sample])
    np.testing.assert_allclose(c, o["conf"], rtol=0, atol=parity.CONF_TOL)
    sure = o["gap"] > parity.GAP_TOL                    # argmax unique beyond 1e-2
    assert np.array_equal(a[sure], o["idx"][sure])
    return o


@pytest.mark.parametrize("V,H,P", [
    (4096, 256, 16),
    (1000, 128, 33),        # ragged last tile (V % 128 = 104), M not a multiple of 16
    (2112, 192, 256),       # M = 256 (one full MMA chunk), V % 128 = 64
    (40000, 512, 256),      # 313 tiles: two or three per CTA, eight K blocks (ring wraps)
    (20032, 64, 7),         # V % 128 = 64 with more tiles than CTAs, a single K block
])
def test_static_head_matches_oracle_and_context_path_on_two_calls(V, H, P):
    cai.cai_test_head_grid_limit(0)
    W = synth.lm_head_weight(V, H, seed=1234, device="cuda")
    wl = synth.Workload("rows", B=1, H=H, V=V, gen_len=P, P=P, T=4, a0="u04")
    hs = synth.HiddenStates(wl, W, "calibrated", seed=21)
    for t in (0, 2):                                  # two calls, different rows
        h = hs(0, t).reshape(P, H).contiguous()
        conf, arg = _static(W, h)
        o = _check_against_oracle(W, h, conf, arg)
        ref_conf, ref_arg = _context_head(W, h, P, H, V)
        np.testing.assert_allclose(conf, ref_conf, rtol=0, atol=parity.CONF_TOL)
        sure = o["gap"] > parity.GAP_TOL
        assert np.array_equal(arg[sure], ref_arg[sure])


@pytest.mark.parametrize("name", ["llada", "dream"])
@pytest.mark.parametrize("M", [32, 256])
def test_static_head_full_size(name, M):
    # V = 126464 / 152064 rows in 988 / 1188 tiles of 128 over the SMs (six to
    # eight tiles per CTA) and H = 4096 / 3584 (64 / 56 K blocks through a
    # four-stage ring): every row against the context path, a sample of rows
    # against the oracle, on two calls in a row.
    wl = synth.WORKLOADS[name]
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device="cuda")
    rows_wl = synth.Workload("rows", B=1, H=wl.H, V=wl.V, gen_len=M, P=M, T=4, a0=wl.a0)
    hs = synth.HiddenStates(rows_wl, W, "calibrated", seed=3)
    rng = np.random.default_rng(M)
    for t in (0, 3):
        h = hs(0, t).reshape(M, wl.H).contiguous()
        conf, arg = _static(W, h)
        sample = np.sort(rng.choice(M, size=min(8, M), replace=False))
        o = _check_against_oracle(W, h, conf, arg, sample)
        ref_conf, ref_arg = _context_head(W, h, M, wl.H, wl.V)
        np.testing.assert_allclose(conf, ref_conf, rtol=0, atol=parity.CONF_TOL)
        assert np.array_equal(arg[sample][o["gap"] > parity.GAP_TOL],
                              ref_arg[sample][o["gap"] > parity.GAP_TOL])


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
    # Host memory is refused before anything is launched: W, rows or an output.
    Wh, rh = W.cpu(), rows[:M].cpu()
    ch, ah = torch.empty((M,), dtype=torch.float32), torch.empty((M,), dtype=torch.int32)
    for args in ((Wh, rows[:M], conf, arg), (W, rh, conf, arg), (W, rows[:M], ch, arg),
                 (W, rows[:M], conf, ah)):
        with pytest.raises(cai.CaiError) as e:
            cai.cai_head_rows_static(*args)
        assert e.value.status == cai.CAI_ERR_ARG
    # The device's free memory does not move across calls (after a first
    # call, which sets the entry point up on this device).
    cai.cai_head_rows_static(W, rows[:M], conf, arg)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for k in range(5):
        cai.cai_head_rows_static(W, rows[k:k + M], conf, arg)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    # The library's own allocator armed to fail: this path never calls it.
    cai.cai_test_fail_alloc_after(1)
    try:
        cai.cai_head_rows_static(W, rows[:M], conf, arg)
        torch.cuda.synchronize()
    finally:
        cai.cai_test_fail_alloc_after(0)
    _check_against_oracle(W, rows[:M], conf[:M].cpu().numpy(), arg[:M].cpu().numpy())


def test_static_head_failed_wait_gives_nan_and_next_call_recovers():
    # A bounded wait that gives up (the hook makes one run out on a barrier
    # nothing arrives at, 2 s) turns that call's outputs into NaN / -1; the
    # error word is then cleared, and the next call is correct again.
    import time
    V, H, M = 4096, 256, 24
    W = synth.lm_head_weight(V, H, device="cuda")
    wl = synth.Workload("rows", B=1, H=H, V=V, gen_len=M, P=M, T=4, a0="u04")
    h = synth.HiddenStates(wl, W, "calibrated", seed=8)(0, 1).reshape(M, H).contiguous()
    cai.cai_test_static_wait_timeout()
    t0 = time.perf_counter()
    conf, arg = _static(W, h)
    assert 1.5 < time.perf_counter() - t0 < 30.0
    assert np.all(np.isnan(conf)) and np.all(arg == -1)
    conf, arg = _static(W, h)
    _check_against_oracle(W, h, conf, arg)
