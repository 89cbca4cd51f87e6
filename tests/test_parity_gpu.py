"""GPU parity: the sm_103a path through the C ABI against the oracle.

Every test here runs the decoding head and commit rule on the GPU (gather,
tcgen05 LM head with the online softmax epilogue, merge + commit) and checks
each step teacher-forced against the fp64 oracle (``tests/parity.py``).
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests import parity

import paper_2608_22646_gb300 as cai

pytestmark = pytest.mark.gpu


def _ctx(B, P, H, V, T, n_blocks, preset=0, flags=None, W=None, seed=1234):
    if W is None:
        W = synth.lm_head_weight(V, H, seed=seed, device="cuda")
    cfg = cai.cai_config_default(preset, B, P, H, V, T, n_blocks)
    if flags is not None:
        cfg.flags = flags
    return cai.cai_init(cfg, W), W


def _wl(name, **kw):
    wl = synth.WORKLOADS[name]
    return synth.Workload(**{**wl.__dict__, **kw})


def test_toy_trajectory_every_step():
    wl = synth.WORKLOADS["toy"]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "calibrated")
    try:
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows > wl.P * wl.n_blocks      # several steps per block
        assert np.all(final["exit_reason"] != 0)
        print(rep)
    finally:
        cai.cai_free(ctx)


def test_toy_literal_generator_grinds_at_t3():
    wl = synth.WORKLOADS["toy"]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "literal")
    try:
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        assert np.all(final["exit_reason"] == cai.CAI_EXIT_GRIND)
        assert np.all(final["exit_step"] == 3)
        assert np.all(final["tok"] == -1)
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("shape,grid", [
    # (B, P, H, V, T, n_blocks), LM-head CTA cap: ragged vocab tails (V % 8,
    # V % 128), a single K stage (H = 64), M = 1, several MMA chunks (M > 256),
    # B P not a multiple of 16, CTAs with several 128-row tiles and a short one.
    ((1, 1, 64, 64, 4, 2), 0),
    ((3, 7, 128, 1000, 6, 2), 0),
    ((3, 7, 128, 1000, 6, 2), 3),
    ((2, 33, 192, 2112, 8, 2), 5),
    ((2, 150, 64, 4160, 5, 1), 0),
    ((2, 150, 64, 4160, 5, 1), 7),
    ((5, 64, 256, 8192, 12, 2), 9),
    ((1, 16, 256, 4096, 8, 4), 1),
    ((2, 5, 128, 1003, 6, 2), 2),
    ((1, 24, 64, 2085, 6, 1), 0),
])
def test_ragged_shapes_trajectory(shape, grid):
    B, P, H, V, T, nb = shape
    wl = synth.Workload("ragged", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    cai.cai_test_head_grid_limit(grid)
    try:
        ctx, W = _ctx(B, P, H, V, T, nb,
                      flags=cai.CAI_GATING | cai.CAI_POS_FACTOR | cai.CAI_QUARTER_POS)
    finally:
        cai.cai_test_head_grid_limit(0)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=7)
    try:
        if grid:
            assert cai.cai_get_stats(ctx)["grid"] == grid
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("preset,flags", [
    (cai.CAI_PRESET_DREAM, None),  # gating OFF: budgets and grinding exit disabled
    (cai.CAI_PRESET_LLADA, cai.CAI_GATING | cai.CAI_POS_FACTOR | cai.CAI_FLUSH_ON_EXIT),
    (cai.CAI_PRESET_LLADA, cai.CAI_GATING | cai.CAI_QUARTER_BLOCKS),
    # ablation rows of the paper's component table: "+APD" (Box 3 alone) and
    # "+APD+Block" (Boxes 3-4), both without budgets or position factors
    (cai.CAI_PRESET_LLADA, cai.CAI_NO_BLOCK_SCHEDULE),
    (cai.CAI_PRESET_LLADA, 0),
])
def test_controller_variants(preset, flags):
    wl = _wl("toy", B=4, a0="bimodal", gen_len=128)
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks, preset=preset, flags=flags)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=3)
    try:
        parity.run_checked_trajectory(ctx, W, hs)
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("theta", [0.9, 0.7])
def test_fixed_threshold_rule(theta):
    # The fixed-threshold rule the paper compares with (Fast-dLLM), on a batch
    # of four and on a multi-kernel context (B P = 320).
    for B, P, gen in ((4, 16, 64), (5, 64, 128)):
        wl = _wl("toy", B=B, P=P, a0="bimodal", gen_len=gen)
        W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
        cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
        cfg.flags = cai.CAI_FIXED_THRESHOLD
        cfg.theta_s = theta
        ctx = cai.cai_init(cfg, W)
        try:
            parity.run_checked_trajectory(ctx, W, synth.HiddenStates(wl, W, "calibrated", seed=5))
        finally:
            cai.cai_free(ctx)


@pytest.mark.parametrize("B,P,gen,env", [
    (2, 16, 64, {}), (5, 64, 128, {}), (2, 16, 64, {"CAI_ROWS_HEAD": "0"}),
    (4, 64, 128, {"CAI_FUSED_MAX_BP": "256"}), (5, 64, 128, {"CAI_PAIR_SWAP": "0"})])
def test_rmsnorm_in_head(B, P, gen, env, monkeypatch):
    # Final RMSNorm folded into the head: single-kernel contexts (B P = 32 on
    # the rows-operand kernel, and on the swapped-operand one; B P = 256 on the
    # swapped-operand one), whose LM head computes the row scales itself, and
    # multi-kernel ones (B P = 320: the gather's scales, pair kernel; with
    # CAI_PAIR_SWAP=0 the swapped-operand kernel takes the narrow steps).
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    wl = _wl("toy", B=B, P=P, a0="bimodal", gen_len=gen)
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    g = synth.final_norm_weight(wl.H, seed=9, device="cuda")
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    ctx = cai.cai_init_rmsnorm(cfg, W, g, 1e-5)
    try:
        hs = synth.HiddenStates(wl, W, "calibrated", seed=13)
        rep, _ = parity.run_checked_trajectory(ctx, W, synth.PreNormHidden(hs, seed=21))
        assert rep.rows >= B * P
    finally:
        cai.cai_free(ctx)


def test_rmsnorm_identity_matches_plain_head():
    # g = 1, eps = 0 on rows of unit mean square: the norm is the identity, so
    # the normed context takes the plain context's decisions step for step.
    wl = _wl("toy", B=2)
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    one = torch.ones(wl.H, dtype=torch.bfloat16, device="cuda")
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    gen_ = torch.Generator(device="cpu").manual_seed(4)
    signs = (torch.randint(0, 2, (wl.T * wl.n_blocks, wl.B, wl.P, wl.H), generator=gen_) * 2 - 1)
    hid = lambda blk, t: (signs[blk * wl.T + t] * 1.0).to(torch.bfloat16).to("cuda")
    a = cai.cai_init(cfg, W)
    b = cai.cai_init_rmsnorm(cfg, W, one, 0.0)
    try:
        for blk in range(wl.n_blocks):
            if blk:
                cai.cai_block_advance(a)
                cai.cai_block_advance(b)
            for t in range(3):
                step = cai.cai_first_step if t == 0 else cai.cai_denoise_step
                step(a, hid(blk, t))
                step(b, hid(blk, t))
                torch.cuda.synchronize()
                sa, sb = cai.cai_state_download(a), cai.cai_state_download(b)
                np.testing.assert_allclose(sa["conf"], sb["conf"], rtol=0, atol=2e-3)
                np.testing.assert_array_equal(sa["cand"], sb["cand"])
                if cai.cai_poll(a, 0, 5000) or cai.cai_poll(b, 0, 5000):
                    break
    finally:
        cai.cai_free(a)
        cai.cai_free(b)


@pytest.mark.parametrize("B,P,gen", [(2, 16, 64), (5, 64, 128)])
def test_diagnostics_stability_and_drift(B, P, gen):
    # Section 2.1 diagnostics on a single- and a multi-kernel context: the
    # stability steps and same-argmax runs bit-exact against the oracle, the
    # drift of every step within 1e-4 relative (checked in parity).
    wl = _wl("toy", B=B, P=P, a0="bimodal", gen_len=gen)
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks,
                  flags=cai.CAI_GATING | cai.CAI_POS_FACTOR | cai.CAI_DIAGNOSTICS)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=31)
    try:
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        assert (final["stable"] >= 2).any()
        assert np.isfinite(final["drift"][:, 0, 1]).all()
    finally:
        cai.cai_free(ctx)


def test_guard_bytes_detect_a_write_past_a_buffer():
    # The guard check itself: a host-issued memset of one byte just past the
    # token buffer (inside its guard region, memory the context owns) must be
    # reported; nothing else is touched.
    import ctypes
    cudart = None
    for name in ("libcudart.so", "libcudart.so.13", "/usr/local/cuda/lib64/libcudart.so"):
        try:
            cudart = ctypes.CDLL(name)
            break
        except OSError:
            continue
    if cudart is None:
        pytest.skip("libcudart not found")
    wl = synth.WORKLOADS["toy"]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    try:
        assert cai.cai_test_check_guards(ctx) == 0
        tok = cai.cai_get_state(ctx)["tok"]
        used = wl.B * wl.n_blocks * wl.P * 4
        padded = (used + 255) // 256 * 256
        cudart.cudaMemset.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t]
        assert cudart.cudaMemset(ctypes.c_void_p(tok + padded), 0, 1) == 0
        assert cai.cai_test_check_guards(ctx) == 1
    finally:
        cai.cai_free(ctx)


def test_fraction_eta_mode():
    wl = _wl("toy", B=2)
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    cfg.eta_mode = 1
    cfg.eta_bar = 0.015
    ctx = cai.cai_init(cfg, W)
    try:
        parity.run_checked_trajectory(ctx, W, synth.HiddenStates(wl, W, "calibrated", seed=11))
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("B", [2, 5])
def test_all_commit_at_step_zero_and_noop_steps(B):
    # Hidden rows equal to a scaled W row make every confidence ~1: every
    # token commits at t = 0, the block exits DONE, and later steps decode
    # nothing.  B P = 32: single-kernel steps; 80: multi-kernel steps, whose
    # pair LM head records the empty step's M = 0 itself.
    P, H, V, T = 16, 256, 4096, 8
    ctx, W = _ctx(B, P, H, V, T, 2)
    try:
        assert (cai.cai_get_stats(ctx)["kernels_per_step"] == 1) == (B * P <= 64)
        tgt = torch.arange(B * P, device="cuda") * 37 % V
        h = (W[tgt].float() * 400.0).to(torch.bfloat16).reshape(B, P, H)
        cai.cai_first_step(ctx, h)
        assert cai.cai_poll(ctx, 0, 5000)
        st = cai.cai_state_download(ctx)
        assert np.array_equal(st["tok"][:, :P].reshape(-1), tgt.cpu().numpy())
        assert np.all(st["exit_reason"][:, 0] == cai.CAI_EXIT_DONE)
        assert np.all(st["exit_step"][:, 0] == 0)
        with pytest.raises(cai.CaiError) as e:      # poll saw the block end
            cai.cai_denoise_step(ctx, h)
        assert e.value.status == cai.CAI_ERR_ORDER
        cai.cai_block_advance(ctx)
        cai.cai_first_step(ctx, h)
        cai.cai_denoise_step(ctx, h)                # issued before a poll: decodes nothing
        torch.cuda.synchronize()
        st = cai.cai_state_download(ctx)
        assert st["m_hist"][1, 0] == B * P and st["m_hist"][1, 1] == 0
    finally:
        cai.cai_free(ctx)


def _expected_kernels(st, rows_cap):
    """Launches per multi-kernel step: gather, merge + commit, the LM head(s),
    and the row merge when some step size leaves per-tile partials."""
    if not st["pair_grid"]:
        return 3
    pairs = st["pair_grid"] // 2
    reduce = any(pairs % rt for rt in range(1, -(-rows_cap // 256) + 1))
    head = st["pair_swap_max_n"] < 32  # the swapped-operand kernel takes M < 32
    return 2 + (1 if head else 0) + 1 + (1 if reduce else 0)


@pytest.mark.parametrize("pair,swap,max_n", [("1", "1", None), ("1", "1", "256"),
                                             ("1", "0", None), ("0", "1", None)])
def test_pair_kernel_steps(pair, swap, max_n, monkeypatch):
    # B P = 320 > 256: multi-kernel steps.  The pair kernel decodes every step,
    # swapped while the tile width is at most 192 (default; 256: always):
    # two row tiles of 160 at M = 320, one narrowing tile below 192 rows, the
    # unswapped 256-row tile in between.  CAI_PAIR_SWAP=0: steps with >= 32
    # masked rows run on the unswapped pair kernel (two 256-row tiles, the
    # second mostly padding), smaller ones on the swapped-operand kernel;
    # CAI_PAIR=0 keeps every step on the latter.
    monkeypatch.setenv("CAI_PAIR", pair)
    monkeypatch.setenv("CAI_PAIR_SWAP", swap)
    if max_n:
        monkeypatch.setenv("CAI_PAIR_SWAP_MAX_N", max_n)
    B, P, H, V, T, nb = 5, 64, 256, 8000, 10, 2
    wl = synth.Workload("pairsteps", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    ctx, W = _ctx(B, P, H, V, T, nb, flags=cai.CAI_GATING | cai.CAI_POS_FACTOR)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=17)
    try:
        st = cai.cai_get_stats(ctx)
        want = (int(max_n or 192) if swap == "1" else 0) if pair == "1" else 0
        assert st["pair_swap_max_n"] == want
        assert st["kernels_per_step"] == _expected_kernels(st, B * P)
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        st = cai.cai_state_download(ctx)
        assert int(st["m_hist"].max()) >= 128   # the pair kernel decoded some steps
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("clusters,max_n,shape", [
    # (pairs, widest swapped tile, (B, P, H, V, T, n_blocks)).  3 pairs: M in
    # (256, 512] has two row tiles, not a divisor of 3, so partials are written
    # per vocabulary tile (and CTA, swapped) and merged by the reduce kernel;
    # M <= 256 and M in (512, 768] keep one partial per pair (and CTA).
    # V % 256 = 184: the odd CTA's half of the last vocabulary tile is partly
    # past V; V % 256 = 84: entirely past V.  H = 64: a single K block.
    # max_n 256: every step swapped; 0: none; 192: both kinds in one
    # trajectory (M = 576: three 192-wide tiles swapped, M ~ 400 unswapped).
    (3, "256", (9, 64, 128, 3000, 10, 1)),
    (3, "0", (9, 64, 128, 3000, 10, 1)),
    (3, "192", (9, 64, 128, 3000, 10, 1)),
    (2, "256", (9, 64, 64, 2900, 8, 1)),
    (1, "256", (6, 50, 192, 4100, 8, 2)),
    (1, "192", (6, 50, 192, 4100, 8, 2)),
])
def test_pair_partial_layouts(clusters, max_n, shape, monkeypatch):
    monkeypatch.setenv("CAI_PAIR_CLUSTERS", str(clusters))
    if max_n == "0":
        monkeypatch.setenv("CAI_PAIR_SWAP", "0")
    else:
        monkeypatch.setenv("CAI_PAIR_SWAP_MAX_N", max_n)
    B, P, H, V, T, nb = shape
    wl = synth.Workload("swaplayouts", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    ctx, W = _ctx(B, P, H, V, T, nb, flags=cai.CAI_GATING | cai.CAI_POS_FACTOR)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=23)
    try:
        st = cai.cai_get_stats(ctx)
        assert st["pair_grid"] == 2 * clusters and st["pair_swap_max_n"] == int(max_n)
        assert st["kernels_per_step"] == _expected_kernels(st, B * P)
        rep, _ = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("shape", [
    # (B, P, H, V, T, n_blocks), all multi-kernel.  B P = 65: one over the
    # single-kernel limit, a 96-wide swapped tile whose odd half runs past the
    # 80-row buffer (TMA fills zeros).  V = 130: the odd CTA's vocabulary half
    # holds 2 rows; V = 128: none.  B P = 287 (buffer 288): the first step's two
    # 160-wide swapped tiles end at row 320.  B P = 400: the first steps run
    # unswapped (224-wide tiles would be needed), later ones swapped.
    (1, 65, 64, 130, 6, 2),
    (3, 22, 128, 128, 6, 2),
    (7, 41, 192, 777, 6, 1),
    (2, 200, 64, 1000, 5, 1),
])
def test_multi_kernel_edge_shapes(shape):
    B, P, H, V, T, nb = shape
    wl = synth.Workload("edges", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    ctx, W = _ctx(B, P, H, V, T, nb, flags=cai.CAI_GATING | cai.CAI_POS_FACTOR)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=37)
    try:
        assert cai.cai_get_stats(ctx)["kernels_per_step"] > 1
        rep, _ = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("ring_max", ["2", "12"])
def test_pair_ring_depths(ring_max, monkeypatch):
    # The pair kernel's ring at its smallest (two stages, every copy waits
    # for the previous stage's MMAs) and largest depth (swapped stages cut to
    # size: up to 10 in flight), over steps of both orientations and of one
    # and two row tiles (B P = 320).
    monkeypatch.setenv("CAI_PAIR_RING_MAX", ring_max)
    B, P, H, V, T, nb = 5, 64, 256, 4096, 8, 2
    wl = synth.Workload("ring", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    ctx, W = _ctx(B, P, H, V, T, nb, flags=cai.CAI_GATING | cai.CAI_POS_FACTOR)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=53)
    try:
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P and int(final["m_hist"].max()) > 256
    finally:
        cai.cai_free(ctx)


def _random_shapes(n, seed=2608):
    rng = np.random.default_rng(seed)
    out = []
    while len(out) < n:
        B = int(rng.integers(1, 13))
        P = int(rng.choice([8, 16, 24, 32, 48, 64]))
        H = int(rng.choice([64, 128, 192, 256]))
        V = int(rng.integers(128, 6000))
        T = int(rng.integers(4, 11))
        nb = int(rng.choice([1, 2]))
        if 8 <= B * P <= 768:
            out.append((B, P, H, V, T, nb))
    return out


@pytest.mark.parametrize("shape", _random_shapes(14))
def test_random_shape_trajectories(shape):
    # Seeded random shapes (mostly multi-kernel: both pair orientations, one to
    # three row tiles, ragged vocabularies and hidden sizes), each a full
    # trajectory checked step by step against the oracle.
    B, P, H, V, T, nb = shape
    wl = synth.Workload("random", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    ctx, W = _ctx(B, P, H, V, T, nb, flags=cai.CAI_GATING | cai.CAI_POS_FACTOR)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=B * 1000 + P)
    try:
        rep, _ = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P
    finally:
        cai.cai_free(ctx)


def test_teacher_forced_random_states():
    # Random mid-block states uploaded into the context, then one step.
    wl = _wl("toy", B=6, P=16, gen_len=32, T=20)
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=5)
    ocfg = parity.oracle_config(ctx.cfg)
    rng = np.random.default_rng(0)
    try:
        for trial in range(6):
            blk = int(rng.integers(0, wl.n_blocks))
            t = int(rng.integers(1, wl.T))
            st = cai.cai_state_download(ctx)
            for k in ("tok", "cstep", "cand", "budget", "conf", "s0"):
                st[k][:] = 0
            st["tok"][:] = -1
            st["cstep"][:] = -1
            sl = slice(blk * wl.P, (blk + 1) * wl.P)
            committed = rng.random((wl.B, wl.P)) < 0.4
            st["tok"][:, sl] = np.where(committed, rng.integers(0, wl.V, (wl.B, wl.P)), -1)
            st["cstep"][:, sl] = np.where(committed, rng.integers(0, t, (wl.B, wl.P)), -1)
            st["budget"][:, sl] = rng.choice([8, 32, 64], (wl.B, wl.P))
            st["ell"][:] = rng.integers(0, 4, wl.B)
            st["exit_reason"][:] = 0
            st["exit_reason"][:, blk] = np.where(rng.random(wl.B) < 0.2, 1, 0)
            st["exit_step"][:] = -1
            st["unresolved"][:] = 0
            st["m_hist"][:] = 0
            st["blk"], st["t_next"] = blk, t
            cai.cai_state_upload(ctx, st)
            pre = cai.cai_state_download(ctx)
            h = hs(blk, t)
            cai.cai_denoise_step(ctx, h)
            torch.cuda.synchronize()
            post = cai.cai_state_download(ctx)
            parity.check_step(ocfg, oracle.bf16_bits(W), h, pre, post, blk, t)
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("shape,host", [("toy", "pinned"), ("toy", "pageable"),
                                        ("multi", "pinned"), ("multi", "pageable")])
def test_host_hidden_and_host_weight_match_device(shape, host):
    # Host inputs: copied on the context's side stream into alternating device
    # buffers (page-locked or pageable memory, single- or multi-kernel steps);
    # a host W is copied once at init.
    wl = synth.WORKLOADS["toy"]
    if shape == "multi":
        wl = _wl("toy", B=5, P=64, gen_len=128)
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    hs = synth.HiddenStates(wl, W, "calibrated")
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    a = cai.cai_init(cfg, W)
    Wh = W.cpu().pin_memory()
    b = cai.cai_init(cfg, Wh)
    try:
        for blk in range(2):
            if blk:
                cai.cai_block_advance(a)
                cai.cai_block_advance(b)
            for t in range(wl.T):
                h = hs(blk, t)
                step = cai.cai_first_step if t == 0 else cai.cai_denoise_step
                step(a, h)
                hh = h.cpu()
                if host == "pinned":
                    hh = hh.pin_memory()
                step(b, hh)
                torch.cuda.synchronize()
                if cai.cai_poll(a, 0, 5000):
                    break
        sa, sb = cai.cai_state_download(a), cai.cai_state_download(b)
        for k in ("tok", "conf", "cand", "exit_reason", "m_hist"):
            assert np.array_equal(sa[k], sb[k]), k
        out = torch.empty((wl.B, wl.n_blocks * wl.P), dtype=torch.int32).pin_memory()
        cai.cai_read_tokens(a, out)
        torch.cuda.synchronize()
        assert np.array_equal(out.numpy(), sa["tok"])
    finally:
        cai.cai_free(a)
        cai.cai_free(b)


@pytest.mark.parametrize("B,host,mode", [(1, "pinned", ""), (2, "pinned", ""),
                                         (2, "pageable", ""), (5, "pinned", ""),
                                         (5, "pageable", ""), (5, "pinned", "norm"),
                                         (5, "pinned", "diag"), (2, "pinned", "norm"),
                                         (5, "pinned", "swap0")])
def test_host_rows_pipelined_match_device(B, host, mode, monkeypatch):
    # Whole trajectories issued back to back with no synchronisation between
    # steps (a one-step-behind poll only), every step reading a different host
    # buffer: the rows are copied on the context's side stream into two
    # alternating buffers while the previous step runs, and the step's first
    # reader (the single-kernel LM head, B <= 2, or the gather, B = 5) waits
    # for the copy on the device; with the final norm in single-kernel steps,
    # or with the diagnostics' drift kernel, the step's stream waits for it
    # instead.  swap0: multi-kernel steps also launch the swapped-operand LM
    # head (CAI_PAIR_SWAP=0), which reads the gathered rows.  The states must
    # equal those of the same trajectory on device inputs bit for bit.
    if mode == "swap0":
        monkeypatch.setenv("CAI_PAIR_SWAP", "0")
    P = 16 if B < 5 else 64
    wl = _wl("toy", B=B, P=P, gen_len=4 * P)
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    hs = synth.HiddenStates(wl, W, "calibrated", seed=29)
    dev_in = [[hs(blk, t) for t in range(wl.T)] for blk in range(wl.n_blocks)]
    host_in = [[(x.cpu().pin_memory() if host == "pinned" else x.cpu().clone()) for x in row]
               for row in dev_in]
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    if mode == "diag":
        cfg.flags |= cai.CAI_DIAGNOSTICS
    if mode == "norm":
        g = synth.final_norm_weight(wl.H).cuda()
        a = cai.cai_init_rmsnorm(cfg, W, g, 1e-5)
        b = cai.cai_init_rmsnorm(cfg, W, g, 1e-5)
    else:
        a = cai.cai_init(cfg, W)
        b = cai.cai_init(cfg, W)
    try:
        for ctx, inp in ((a, dev_in), (b, host_in)):
            for rep in range(2):
                cai.cai_reset(ctx)
                for blk in range(wl.n_blocks):
                    if blk:
                        cai.cai_block_advance(ctx)
                    cai.cai_first_step(ctx, inp[blk][0])
                    for t in range(1, wl.T):
                        if t >= 2 and cai.cai_poll(ctx, 1, 60000):
                            break
                        cai.cai_denoise_step(ctx, inp[blk][t])
            torch.cuda.synchronize()
        sa, sb = cai.cai_state_download(a), cai.cai_state_download(b)
        keys = ["tok", "conf", "cand", "cstep", "exit_reason", "exit_step", "m_hist"]
        if mode == "diag":
            keys += ["stable", "drift"]
        for k in keys:
            assert np.array_equal(sa[k], sb[k], equal_nan=(k == "drift")), k
        assert int(sa["m_hist"].sum()) > 0
        assert cai.cai_test_check_guards(b) == 0
    finally:
        cai.cai_free(a)
        cai.cai_free(b)


def test_device_wait_timeout_reports_and_device_stays_usable():
    # A kernel waits, through the step kernels' bounded barrier wait, on a
    # barrier nothing arrives at: after the limit it records the failure in
    # the context's error word and returns.  The host then reads
    # CAI_ERR_DEVICE, the context stays sticky (its device error word names
    # the wait that gave up), and a new context on the same GPU runs a checked
    # trajectory.
    import time
    wl = synth.WORKLOADS["toy"]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=41)
    try:
        cai.cai_first_step(ctx, hs(0, 0))
        torch.cuda.synchronize()
        cai.cai_state_download(ctx)                      # healthy so far
        t0 = time.perf_counter()
        cai.cai_test_wait_timeout(ctx)
        torch.cuda.synchronize()
        assert 1.5 < time.perf_counter() - t0 < 30.0     # the wait ran to its limit
        assert cai.cai_device_error_bits(ctx) == (1 << cai.DEVERR_NAMES.index("wait_full"))
        with pytest.raises(cai.CaiError) as e:
            cai.cai_state_download(ctx)
        assert e.value.status == cai.CAI_ERR_DEVICE
        assert cai.cai_device_error_bits(ctx) == (1 << cai.DEVERR_NAMES.index("wait_full"))
        with pytest.raises(cai.CaiError) as e:
            cai.cai_denoise_step(ctx, hs(0, 1))
        assert e.value.status == cai.CAI_ERR_DEVICE
    finally:
        cai.cai_free(ctx)
    ctx2, W2 = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    try:
        parity.run_checked_trajectory(ctx2, W2, synth.HiddenStates(wl, W2, "calibrated", seed=43))
    finally:
        cai.cai_free(ctx2)


@pytest.mark.parametrize("B,P", [(2, 16), (5, 64)])
def test_checkpoint_resume_in_new_context(B, P):
    # Checkpoint/resume: a trajectory interrupted after a few steps of its
    # second block, its state downloaded, freed, uploaded into a new context
    # and continued, ends exactly where the uninterrupted trajectory does.
    wl = _wl("toy", B=B, P=P, gen_len=3 * P, a0="bimodal")
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    hs = synth.HiddenStates(wl, W, "calibrated", seed=47)
    inp = [[hs(blk, t) for t in range(wl.T)] for blk in range(wl.n_blocks)]
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)

    def run(ctx, start_blk=0, start_t=0, stop=None):
        for blk in range(start_blk, wl.n_blocks):
            if blk > start_blk or (blk == start_blk and start_t == 0 and blk > 0):
                cai.cai_block_advance(ctx)
            for t in range(start_t if blk == start_blk else 0, wl.T):
                if stop == (blk, t):
                    torch.cuda.synchronize()
                    return
                (cai.cai_first_step if t == 0 else cai.cai_denoise_step)(ctx, inp[blk][t])
                torch.cuda.synchronize()
                if cai.cai_poll(ctx, 0, 5000):
                    break
        torch.cuda.synchronize()

    a = cai.cai_init(cfg, W)
    try:
        run(a)
        full = cai.cai_state_download(a)
    finally:
        cai.cai_free(a)
    b = cai.cai_init(cfg, W)
    try:
        run(b, stop=(1, 2))
        ckpt = cai.cai_state_download(b)
    finally:
        cai.cai_free(b)
    assert ckpt["blk"] == 1 and ckpt["t_next"] == 2
    c = cai.cai_init(cfg, W)
    try:
        cai.cai_state_upload(c, ckpt)
        run(c, start_blk=1, start_t=2)
        resumed = cai.cai_state_download(c)
    finally:
        cai.cai_free(c)
    for k in ("tok", "conf", "cand", "cstep", "budget", "s0", "exit_reason", "exit_step",
              "unresolved", "m_hist"):
        assert np.array_equal(full[k], resumed[k]), k


def test_order_errors_and_poll():
    wl = synth.WORKLOADS["toy"]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, 2)
    hs = synth.HiddenStates(wl, W, "calibrated")
    try:
        h = hs(0, 0)
        with pytest.raises(cai.CaiError) as e:        # misaligned hidden pointer
            cai.cai_first_step(ctx, h.data_ptr() + 2)
        assert e.value.status == cai.CAI_ERR_ARG
        for fn in (lambda: cai.cai_denoise_step(ctx, h), lambda: cai.cai_block_advance(ctx)):
            with pytest.raises(cai.CaiError) as e:
                fn()
            assert e.value.status == cai.CAI_ERR_ORDER
        assert not cai.cai_poll(ctx, 0, 100)          # nothing issued yet
        cai.cai_first_step(ctx, h)
        with pytest.raises(cai.CaiError) as e:
            cai.cai_first_step(ctx, h)
        assert e.value.status == cai.CAI_ERR_ORDER
        for t in range(1, wl.T):
            cai.cai_denoise_step(ctx, hs(0, t))
        with pytest.raises(cai.CaiError) as e:        # t would reach T
            cai.cai_denoise_step(ctx, h)
        assert e.value.status == cai.CAI_ERR_ORDER
        assert cai.cai_poll(ctx, 0, 5000)             # t = T - 1 always ends the block
        cai.cai_block_advance(ctx)
        cai.cai_first_step(ctx, h)
        with pytest.raises(cai.CaiError) as e:        # already at the last block
            cai.cai_block_advance(ctx)
        assert e.value.status == cai.CAI_ERR_ORDER
    finally:
        cai.cai_free(ctx)


def test_alloc_failure_injection_leaks_nothing():
    wl = synth.WORKLOADS["toy"]
    W = synth.lm_head_weight(wl.V, wl.H, device="cuda")
    cfg = cai.cai_config_default(0, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for n in (1, 5, 12, 20):
        cai.cai_test_fail_alloc_after(n)
        with pytest.raises(cai.CaiError) as e:
            cai.cai_init(cfg, W)
        assert e.value.status == cai.CAI_ERR_NOMEM
    cai.cai_test_fail_alloc_after(0)
    ctx = cai.cai_init(cfg, W)
    cai.cai_free(ctx)
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) < (8 << 20)


def test_profile_and_stats():
    wl = synth.WORKLOADS["toy"]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "calibrated")
    try:
        cai.cai_profile(ctx, True)
        cai.cai_first_step(ctx, hs(0, 0))
        cai.cai_denoise_step(ctx, hs(0, 1))
        s = cai.cai_get_stats(ctx)
        assert s["steps"] == 2 and s["head_launches"] == 2
        assert s["kernels_per_step"] == 1 and s["launches"] == 2    # B P = 16: one kernel
        assert s["head_profiled"] == 2 and s["head_ms"] > 0
        assert s["grid"] == 64 and s["n_max"] == 16
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("name", ["llada", "dream"])
def test_full_size_first_step_sampled(name):
    # Full LLaDA/Dream shapes: one step-zero decode of the whole block, then
    # the oracle recomputes a sample of positions one by one.
    wl = synth.WORKLOADS[name]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "calibrated")
    try:
        h = hs(0, 0)
        cai.cai_first_step(ctx, h)
        torch.cuda.synchronize()
        st = cai.cai_state_download(ctx)
        sample = [0, 5, 17, wl.P - 1]
        rows = oracle.bf16_bits(h.reshape(-1, wl.H))[sample]
        o = oracle.head_rows(W, rows)
        for k, p in enumerate(sample):
            assert abs(st["s0"][0, p] - o["conf"][k]) <= parity.CONF_TOL
            if o["gap"][k] > parity.GAP_TOL:
                assert st["cand"][0, p] == o["idx"][k]
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("name,n_blocks", [("llada", None), ("dream", None)])
def test_full_size_trajectory_every_row(name, n_blocks):
    # The B = 1 configurations at full size (P = 32, the LLaDA or Dream weight
    # shape, single-kernel steps, the calibrated generator): every step of the
    # whole generation (all eight blocks) is checked teacher-forced on every
    # masked row, confidences, argmaxes and every integer field of the state.
    wl = synth.WORKLOADS[name]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks, preset=cai.CAI_PRESET_LLADA)
    hs = synth.HiddenStates(wl, W, "calibrated")
    try:
        assert cai.cai_get_stats(ctx)["kernels_per_step"] == 1
        rep, st = parity.run_checked_trajectory(ctx, W, hs, n_blocks=n_blocks)
        blocks = wl.n_blocks if n_blocks is None else n_blocks
        assert rep.rows >= blocks * wl.P
        assert np.all(st["exit_reason"][:, :blocks] != 0)
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("name,B,P,T,nb,a0", [
    ("b64", 64, 32, 32, 8, "u04"),      # batched LLaDA layout: 2048 rows at step zero
    ("long", 8, 64, 64, 16, "long"),    # long-Dream layout: 16 blocks of 64, T = 64
])
def test_batch_layouts_full_trajectory_small_vocab(name, B, P, T, nb, a0):
    # The batched-LLaDA (B = 64, P = 32, 8 blocks) and long-Dream (B = 8,
    # P = 64, T = 64, 16 blocks, later blocks easier) layouts with a small
    # vocabulary and hidden size, so that the oracle recomputes every row:
    # every step of the whole generation teacher-forced, every field.  At
    # B = 64 the commit kernel runs 64 CTAs and builds the 2048-token row list
    # in four rounds; the long layout runs theta_e^(b) down to its floor
    # (b > 4) and exits blocks early.
    V, H = 4096, 256
    wl = synth.Workload(name, B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0=a0)
    ctx, W = _ctx(B, P, H, V, T, nb)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=B + P)
    try:
        assert cai.cai_get_stats(ctx)["kernels_per_step"] > 1
        rep, final = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P * nb
        assert final["m_hist"][0, 0] == B * P
        assert np.all(final["exit_reason"] != 0)
        ex = final["exit_step"]
        assert (ex < T - 1).all(axis=0).any()          # some block ended early for everyone
        if nb > 4:
            ocfg = parity.oracle_config(ctx.cfg)
            assert oracle.theta_e(ocfg, nb) == pytest.approx(0.40)
            assert (final["exit_reason"][:, 4:] != 0).all()
        print(name, rep, "steps per block", (ex.max(axis=0) + 1).tolist())
    finally:
        cai.cai_free(ctx)


@pytest.mark.parametrize("name", ["llada_batched", "dream_long"])
def test_full_size_batch_trajectory_controller_and_sampled_rows(name):
    # The batched LLaDA (B = 64, H = 4096, V = 126464) and long Dream (B = 8,
    # P = 64, T = 64, H = 3584, V = 152064, 16 blocks) configurations at full
    # size, the whole generation: every step checked at the controller level
    # (the oracle runs Algorithm 1 from the GPU's pre-step state on the GPU's
    # confidences and argmaxes; tokens, commit steps, budgets, low-yield
    # counters, exits and M_t bit-exact), and at step zero of every block
    # plus four seeded steps among each block's others, 14 sampled masked rows
    # (the first and last included) recomputed by the fp64 oracle.
    wl = synth.WORKLOADS[name]
    ctx, W = _ctx(wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    hs = synth.HiddenStates(wl, W, "calibrated")
    seen = set()

    def on_step(blk, t, M):
        seen.add("pair2" if M > 256 else "pair1" if M >= 32 else "narrow" if M else "empty")

    try:
        final = parity.run_controller_checked_trajectory(ctx, W, hs, 4, 12, seed=7,
                                                         on_step=on_step)
        assert np.all(final["exit_reason"] != 0)
        assert final["m_hist"][0, 0] == wl.B * wl.P
        assert {"pair2", "pair1", "narrow"} <= seen, seen
        print(name, "steps per block", (final["exit_step"].max(axis=0) + 1).tolist(),
              "exits", np.bincount(final["exit_reason"].reshape(-1), minlength=4).tolist())
    finally:
        cai.cai_free(ctx)


def test_debug_build_range_checks_stay_quiet():
    # The CAI_DEBUG build checks index lists and partial offsets before every
    # use (a value out of range sets an error bit and the access is skipped).
    # Single- and multi-kernel trajectories run clean on it; any flagged
    # access would surface as CAI_ERR_DEVICE in the state download.
    import os
    import subprocess
    import sys
    from paper_2608_22646_gb300 import build as cai_build
    lib = cai_build.build(debug=True)
    code = (
        "import synth, torch, paper_2608_22646_gb300 as cai\n"
        "from tests import parity\n"
        "for B, P, gen in ((1, 16, 64), (5, 64, 128)):\n"
        "    wl = synth.Workload('dbg', B=B, H=256, V=4096, gen_len=gen, P=P, T=8, a0='u04')\n"
        "    W = synth.lm_head_weight(wl.V, wl.H, device='cuda')\n"
        "    cfg = cai.cai_config_default(0, B, P, wl.H, wl.V, wl.T, wl.n_blocks)\n"
        "    ctx = cai.cai_init(cfg, W)\n"
        "    assert cai.LIB_PATH.endswith('libcai_debug.so')\n"
        "    parity.run_checked_trajectory(ctx, W, synth.HiddenStates(wl, W, 'calibrated', seed=2))\n"
        "    cai.cai_free(ctx)\n"
        "print('debug build clean')\n")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, "-c", code], cwd=root, env={**os.environ, "CAI_LIB": lib},
                         capture_output=True, text=True, timeout=900)
    assert out.returncode == 0, out.stdout[-2000:] + out.stderr[-2000:]
    assert "debug build clean" in out.stdout


def test_bench_json_line_contract():
    # The benchmark's own arm on the toy shape: one JSON line with the
    # contract's keys, a device-timed value, the roofline object, the
    # end-to-end figure through host buffers, clocks and the launch count.
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, "bench.py", "--workload", "toy", "--steps", "3",
                          "--warmup", "3", "--no-cpu-baseline"], cwd=root, capture_output=True,
                         text=True, timeout=900)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "roofline", "e2e", "gpu_launches", "clocks"):
        assert k in line, k
    assert line["value"] > 0 and line["steps"] == 3 and line["warmup"] == 3 and line["n_gpus"] == 1
    assert line["config"]["workload"].startswith("toy")
    roof = line["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in roof, k
    assert abs(roof["frac"] - roof["achieved"] / roof["peak"]) < 1e-3
    e2e = line["e2e"]
    assert e2e["value"] > 0 and e2e["unit"] == line["unit"] and e2e["h2d_bytes_per_step"] > 0
    assert e2e["d2h_bytes_per_step"] > 0
    assert line["gpu_launches"] > 0
    assert line["clocks"]["sm_max_mhz"] > 0


@pytest.mark.parametrize("rows_head,max_bp,shape", [
    # (CAI_ROWS_HEAD, CAI_FUSED_MAX_BP, (B, P, H, V, T, n_blocks)): single-kernel
    # steps of up to 128 rows on the rows-operand LM head (2 to 4 epilogue
    # warps with rows; rows stages of 8 and 16 KiB), ragged V (V % 8, V % 256),
    # one K block (H = 64); and the swapped-operand kernel that CAI_ROWS_HEAD=0
    # selects, at B P <= 32.
    ("1", "64", (2, 32, 256, 4096, 8, 2)),
    ("1", "128", (4, 32, 192, 5003, 8, 2)),
    ("1", "128", (1, 100, 64, 2085, 6, 1)),
    ("1", "32", (1, 20, 128, 300, 6, 2)),
    ("0", "32", (1, 16, 256, 4096, 8, 4)),
    ("0", "32", (2, 16, 128, 1003, 6, 2)),
])
def test_single_kernel_heads(rows_head, max_bp, shape, monkeypatch):
    monkeypatch.setenv("CAI_ROWS_HEAD", rows_head)
    monkeypatch.setenv("CAI_FUSED_MAX_BP", max_bp)
    B, P, H, V, T, nb = shape
    wl = synth.Workload("fused", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    ctx, W = _ctx(B, P, H, V, T, nb, flags=cai.CAI_GATING | cai.CAI_POS_FACTOR)
    hs = synth.HiddenStates(wl, W, "calibrated", seed=B * 31 + P)
    try:
        st = cai.cai_get_stats(ctx)
        assert st["kernels_per_step"] == 1
        assert st["head_rows"] == (1 if rows_head == "1" else 0)
        rep, _ = parity.run_checked_trajectory(ctx, W, hs)
        assert rep.rows >= B * P
    finally:
        cai.cai_free(ctx)
