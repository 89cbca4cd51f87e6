"""Pins of the oracle against facts that do not come from the oracle itself.

Each function of ``oracle`` is checked against at least one of: values printed
in the paper (Boxes 4-6, arXiv 2608.22646), values worked out by hand from the
printed formulas (``tests/golden``), closed forms, high-precision brute force
(mpmath) on tiny inputs, invariants, and hand-worked controller trajectories
that exercise every branch of Algorithm 1.

Coverage map (function -> pins):
  cai_o_bf16_to_double     -> exact bit patterns (test_bf16_decode)
  cai_o_head_rows          -> mpmath brute force, V=2 closed form, uniform,
                              one-hot gap closed form, ties, sum-to-one,
                              c = exp(m - LSE), transposed-operand catch
  cai_o_theta_e            -> Box 4 printed values, floor, quarter mode
  cai_o_theta_block        -> hand-worked golden table, endpoints, monotone
  cai_o_pos_factor         -> Box 6 printed tiers, quarter mode
  cai_o_theta_token        -> clip bounds
  cai_o_budget             -> Box 5 hand table, boundaries
  cai_o_low_yield          -> count and fraction readings
  cai_o_controller_step    -> hand trajectories G1, G2, budget force,
                              DONE, T-exhausted, flush, gating OFF, the
                              low-yield reset at each block's step zero, and
                              invariants over synthetic trajectories
  head_rows_shard,         -> equal to the full-vocabulary head for several
  merge_shards                partitions, a tie across a shard boundary,
                              the two-row closed form
"""
import math
import os

import mpmath
import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    out = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                out.append(line.split())
    return out


def bf16_from_float(x):
    """Round-to-nearest-even float32 -> bf16 bits (test-side helper)."""
    a = np.asarray(x, np.float32).reshape(-1)
    u = a.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    return r.reshape(np.shape(x))


# ------------------------------------------------------------------ bf16 --

def test_bf16_decode():
    lib = oracle.lib()
    assert lib.cai_o_bf16_to_double(0x3F80) == 1.0
    assert lib.cai_o_bf16_to_double(0xC000) == -2.0
    assert lib.cai_o_bf16_to_double(0x3F81) == 1.0 + 2.0 ** -7
    assert lib.cai_o_bf16_to_double(0x0001) == 2.0 ** -133          # smallest subnormal
    assert lib.cai_o_bf16_to_double(0x8000) == 0.0
    assert math.isinf(lib.cai_o_bf16_to_double(0x7F80))
    assert lib.cai_o_bf16_to_double(0x4049) == 3.140625


# ------------------------------------------------------------------ head --

def _brute(Wf, hf):
    """mpmath (60 digits) logits, softmax, confidence, lowest-index argmax."""
    mpmath.mp.dps = 60
    V, H = Wf.shape
    z = [mpmath.fsum(mpmath.mpf(float(Wf[v, k])) * mpmath.mpf(float(hf[k])) for k in range(H))
         for v in range(V)]
    m = max(z)
    idx = min(v for v in range(V) if z[v] == m)
    S = mpmath.fsum(mpmath.e ** (zv - m) for zv in z)
    return [float(zv) for zv in z], float(1 / S), idx, float(m + mpmath.log(S))


@pytest.mark.parametrize("seed", range(12))
def test_head_bruteforce_tiny(seed):
    rng = np.random.default_rng(seed)
    V = int(rng.integers(2, 9))
    H = int(rng.integers(1, 5))
    Wf = rng.normal(0, 1.5, (V, H)).astype(np.float32)
    hf = rng.normal(0, 1.5, (H,)).astype(np.float32)
    Wb, hb = bf16_from_float(Wf), bf16_from_float(hf)
    Wd = Wb.astype(np.uint32) << 16
    hd = hb.astype(np.uint32) << 16
    Wq = Wd.view(np.float32).reshape(V, H)
    hq = hd.view(np.float32)
    z_ref, c_ref, idx_ref, lse_ref = _brute(Wq, hq)
    out = oracle.head_rows(Wb, hb.reshape(1, H))
    assert out["idx"][0] == idx_ref
    assert abs(out["conf"][0] - c_ref) < 1e-13
    assert abs(out["lse"][0] - lse_ref) < 1e-12
    z, p, idx = oracle.softmax_row(Wb, hb)
    np.testing.assert_allclose(z, z_ref, rtol=0, atol=1e-12)
    assert abs(p.sum() - 1.0) < 1e-12
    assert idx == idx_ref


def _q(x):
    """float32 array -> (bf16 bits, the exact float values they decode to)."""
    b = bf16_from_float(np.asarray(x, np.float32))
    return b, (b.astype(np.uint32) << 16).view(np.float32).reshape(np.shape(x))


@pytest.mark.parametrize("seed", range(8))
def test_head_rmsnorm_bruteforce_tiny(seed):
    # The final RMSNorm in the head: x = g h / sqrt(mean h^2 + eps), z = W x,
    # in 60-digit arithmetic on tiny random inputs.
    rng = np.random.default_rng(100 + seed)
    V, H = int(rng.integers(2, 9)), int(rng.integers(1, 6))
    Wb, Wq = _q(rng.normal(0, 1.5, (V, H)))
    hb, hq = _q(rng.normal(0, 2.0, (H,)))
    gb, gq = _q(rng.normal(1, 0.3, (H,)))
    eps = float(rng.choice([0.0, 1e-6, 0.3]))
    mpmath.mp.dps = 60
    r = mpmath.sqrt(mpmath.fsum(mpmath.mpf(float(v)) ** 2 for v in hq) / H + mpmath.mpf(eps))
    x = [mpmath.mpf(float(gq[k])) * mpmath.mpf(float(hq[k])) / r for k in range(H)]
    z = [mpmath.fsum(mpmath.mpf(float(Wq[v, k])) * x[k] for k in range(H)) for v in range(V)]
    m = max(z)
    idx = min(v for v in range(V) if z[v] == m)
    c = float(1 / mpmath.fsum(mpmath.e ** (zv - m) for zv in z))
    out = oracle.head_rows(Wb, hb.reshape(1, H), norm_weight=gb, eps=eps)
    assert out["idx"][0] == idx
    assert abs(out["conf"][0] - c) < 1e-12


def test_head_rmsnorm_reductions():
    rng = np.random.default_rng(7)
    V, H = 41, 64
    Wb, Wq = _q(rng.normal(0, 0.5, (V, H)))
    h = np.where(rng.random((3, H)) < 0.5, -1.0, 1.0)  # mean square exactly 1
    hb, _ = _q(h)
    one, _ = _q(np.ones(H))
    plain = oracle.head_rows(Wb, hb)
    # g = 1, eps = 0 and unit mean square: the norm is the identity
    same = oracle.head_rows(Wb, hb, norm_weight=one, eps=0.0)
    np.testing.assert_array_equal(same["idx"], plain["idx"])
    np.testing.assert_allclose(same["conf"], plain["conf"], rtol=1e-15, atol=0)
    # scale invariance (eps = 0): 2h and h/4 are exact in bf16
    for s in (2.0, 0.25):
        hs, _ = _q(h * s)
        o = oracle.head_rows(Wb, hs, norm_weight=one, eps=0.0)
        np.testing.assert_allclose(o["conf"], plain["conf"], rtol=1e-15, atol=0)
        np.testing.assert_array_equal(o["idx"], plain["idx"])
    # the weight scales the k-th input, not the v-th output: with powers of
    # two, W g is exact in bf16 and the normed head equals the plain head on W g
    gpow = 2.0 ** rng.integers(-2, 3, H)
    gb, _ = _q(gpow)
    Wg, _ = _q(Wq * gpow[None, :])
    folded = oracle.head_rows(Wg, hb)
    normed = oracle.head_rows(Wb, hb, norm_weight=gb, eps=0.0)
    np.testing.assert_array_equal(normed["idx"], folded["idx"])
    np.testing.assert_allclose(normed["conf"], folded["conf"], rtol=1e-14, atol=0)
    # eps, closed form on V = 2: c = sigmoid(|z0 - z1| / sqrt(1 + eps))
    W2b, W2q = _q(rng.normal(0, 0.3, (2, H)))
    for eps in (0.0, 0.5, 3.0):
        o = oracle.head_rows(W2b, hb[:1], norm_weight=one, eps=eps)
        d = abs(float(np.dot(W2q[0].astype(np.float64) - W2q[1], h[0]))) / math.sqrt(1 + eps)
        assert abs(o["conf"][0] - 1.0 / (1.0 + math.exp(-d))) < 1e-14


def test_head_transposed_operand_is_caught():
    # W is deliberately non-square and asymmetric: z = W h differs from any
    # use of W's columns.  h picks column 1 only, so z_v = W[v, 1].
    W = np.array([[1, 2, 0], [3, -4, 0], [0, 8, 1], [5, 6, 7]], np.float32)
    h = np.array([0, 1, 0], np.float32)
    out = oracle.head_rows(bf16_from_float(W), bf16_from_float(h).reshape(1, 3))
    assert out["idx"][0] == 2          # max of column 1 = 8 at row 2
    assert abs(out["zmax"][0] - 8.0) < 1e-15
    assert abs(out["gap"][0] - 2.0) < 1e-15   # 8 - 6


@pytest.mark.parametrize("delta", [0.0, 0.3, 1.0, 4.0, 9.5])
def test_head_two_way_closed_form(delta):
    # V = 2: c = sigma(|z1 - z2|).
    W = np.array([[1.0], [0.0]], np.float32)
    h = np.array([delta], np.float32)
    Wb, hb = bf16_from_float(W), bf16_from_float(h)
    d = float((hb.astype(np.uint32) << 16).view(np.float32)[0])
    out = oracle.head_rows(Wb, hb.reshape(1, 1))
    assert abs(out["conf"][0] - 1.0 / (1.0 + math.exp(-abs(d)))) < 1e-15
    assert out["idx"][0] == 0


@pytest.mark.parametrize("V", [3, 17, 1000])
def test_head_uniform_and_ties(V):
    # All logits equal: c = 1/V and the argmax is the lowest index.
    W = np.ones((V, 4), np.float32)
    h = np.full((4,), 0.5, np.float32)
    out = oracle.head_rows(bf16_from_float(W), bf16_from_float(h).reshape(1, 4))
    assert abs(out["conf"][0] - 1.0 / V) < 1e-15
    assert out["idx"][0] == 0
    assert out["gap"][0] == 0.0


@pytest.mark.parametrize("V,win,delta", [(10, 7, 2.0), (4096, 4095, 5.0), (64, 0, 0.75)])
def test_head_one_hot_gap(V, win, delta):
    # One logit raised by delta above V-1 equal ones: c = 1 / (1 + (V-1) e^-delta).
    W = np.zeros((V, 1), np.float32)
    W[win, 0] = 1.0
    h = np.array([delta], np.float32)
    out = oracle.head_rows(bf16_from_float(W), bf16_from_float(h).reshape(1, 1))
    assert out["idx"][0] == win
    assert abs(out["conf"][0] - 1.0 / (1.0 + (V - 1) * math.exp(-delta))) < 1e-14


def test_head_invariants_random():
    rng = np.random.default_rng(5)
    V, H, M = 300, 64, 6
    W = bf16_from_float(rng.normal(0, 0.3, (V, H)))
    R = bf16_from_float(rng.normal(0, 1.0, (M, H)))
    out = oracle.head_rows(W, R, n_threads=3)
    for i in range(M):
        z, p, idx = oracle.softmax_row(W, R[i])
        assert abs(p.sum() - 1.0) < 1e-12
        assert idx == out["idx"][i]
        assert abs(out["conf"][i] - p.max()) < 1e-15
        assert abs(out["conf"][i] - math.exp(out["zmax"][i] - out["lse"][i])) < 1e-13
        s = np.sort(z)
        assert abs(out["gap"][i] - (s[-1] - s[-2])) < 1e-12
    # thread count does not change any bit
    out1 = oracle.head_rows(W, R, n_threads=1)
    for k in out:
        np.testing.assert_array_equal(out[k], out1[k])


# ------------------------------------------------------------ thresholds --

def test_theta_e_printed_values():
    cfg = oracle.Config()
    for b, te in _rows("block_end_thresholds.txt"):
        assert abs(oracle.theta_e(cfg, int(b)) - float(te)) < 1e-12
    # floor for b > 4 (non-increasing, never below the b = 4 value)
    vals = [oracle.theta_e(cfg, b) for b in range(1, 17)]
    assert all(vals[i + 1] <= vals[i] for i in range(15))
    assert min(vals) == pytest.approx(0.40, abs=1e-12)
    # quarter mode over 16 blocks: blocks 1-4 -> 0.70, 5-8 -> 0.60, 9-12 -> 0.50, 13-16 -> 0.40
    q = oracle.Config(n_blocks=16, flags=oracle.GATING | oracle.POS_FACTOR | oracle.QUARTER_BLOCKS)
    assert [round(oracle.theta_e(q, b), 12) for b in (1, 4, 5, 8, 9, 12, 13, 16)] == \
        [0.7, 0.7, 0.6, 0.6, 0.5, 0.5, 0.4, 0.4]


def test_theta_block_golden():
    for T, b, t, th in _rows("theta_schedule.txt"):
        cfg = oracle.Config(T=int(T))
        assert abs(oracle.theta_block(cfg, int(b), int(t)) - float(th)) < 6e-7, (T, b, t)


@pytest.mark.parametrize("T", [8, 20, 32, 64])
@pytest.mark.parametrize("b", [1, 2, 4, 7])
def test_theta_block_shape(T, b):
    cfg = oracle.Config(T=T, n_blocks=8)
    te = oracle.theta_e(cfg, b)
    th = [oracle.theta_block(cfg, b, t) for t in range(T)]
    assert all(th[i + 1] <= th[i] + 1e-15 for i in range(T - 1))
    assert all(te < x <= 0.9 + 1e-15 for x in th)
    # warm-up: exactly the steps with t < 0.15 T hold theta_s
    for t in range(T):
        assert (th[t] == 0.9) == (t < 0.15 * T) or (t >= 0.15 * T and abs(th[t] - 0.9) < 1e-3)
    # continuity at wT and the end point theta_e at t = T (cosine of pi)
    wT = 0.15 * T
    alpha = (0.9 - te) / 2
    # the first post-warm-up step sits within alpha*(pi*u)^2/2 of theta_s
    t1 = math.ceil(wT)
    u1 = (t1 - wT) / (T - wT)
    assert 0.9 - th[t1] <= alpha * (math.pi * u1) ** 2 / 2 + 1e-12
    # extrapolating one step past T - 1 lands on theta_e to first order
    uL = (T - 1 - wT) / (T - wT)
    assert th[T - 1] - te <= alpha * (math.pi * (1 - uL)) ** 2 / 2 + 1e-12


def test_ablation_variants_thresholds():
    # Box 3 alone ("APD" row of the ablation table): every block follows the
    # block-1 schedule of the golden table (theta_e = 0.70), not Box 4's.
    apd = oracle.Config(T=32, n_blocks=8, flags=oracle.NO_BLOCK_SCHEDULE)
    for T, b, t, th in _rows("theta_schedule.txt"):
        if int(b) != 1:
            continue
        cfg = oracle.Config(T=int(T), n_blocks=8, flags=oracle.NO_BLOCK_SCHEDULE)
        for blk in (1, 2, 4, 8):
            assert abs(oracle.theta_block(cfg, blk, int(t)) - float(th)) < 6e-7, (T, blk, t)
    assert all(oracle.theta_e(apd, b) == pytest.approx(0.70, abs=1e-15) for b in range(1, 9))
    # the fixed-threshold rule the paper compares with (Fast-dLLM): theta_s at
    # every step of every block, position factors still applied when enabled
    for ts in (0.9, 0.7):
        fx = oracle.Config(T=32, P=64, n_blocks=8, theta_s=ts, flags=oracle.FIXED_THRESHOLD)
        assert {oracle.theta_block(fx, b, t) for b in range(1, 9) for t in range(32)} == {ts}
        assert oracle.theta_token(fx, 5, 31, 63) == ts
        fxp = oracle.Config(T=32, P=64, n_blocks=8, theta_s=ts,
                            flags=oracle.FIXED_THRESHOLD | oracle.POS_FACTOR)
        assert oracle.theta_token(fxp, 3, 20, 0) == pytest.approx(ts * 0.8, abs=1e-15)
        assert oracle.theta_token(fxp, 3, 20, 60) == pytest.approx(min(ts * 1.1, 0.98), abs=1e-15)


def test_fixed_threshold_trajectory_commits_exactly_above_threshold():
    # With the fixed rule, gating off and no position factor, a token commits
    # at step t iff its confidence is >= theta_s: check every step of a toy
    # trajectory against the step's own confidences.
    wl = synth.WORKLOADS["toy"]
    cfg = oracle.Config(B=1, P=wl.P, T=wl.T, n_blocks=wl.n_blocks, theta_s=0.7,
                        flags=oracle.FIXED_THRESHOLD)
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device="cpu")
    hs = synth.HiddenStates(wl, W, "calibrated")
    Wb = oracle.bf16_bits(W)
    st = oracle.State(cfg)
    for blk in range(wl.n_blocks):
        for t in range(wl.T):
            before = st.tok.copy()
            out = oracle.step(st, Wb, oracle.bf16_bits(hs(blk, t)), blk, t, 2)
            sl = slice(blk * wl.P, (blk + 1) * wl.P)
            was = before[0, sl] == oracle.MASK
            now = st.tok[0, sl] != oracle.MASK
            conf = st.conf[0, sl]
            assert np.array_equal(now & was, was & (conf >= 0.7)), (blk, t)
            if st.exit_reason[0, blk] != oracle.RUNNING:
                break


def test_drift_closed_forms():
    # Eq. relative_drift on rows whose norms are exact: equal -> 0, doubled ->
    # 1, negated -> 2, orthogonal unit rows -> sqrt(2); the mean over positions.
    H = 16
    e = np.eye(H, dtype=np.float32)
    prev_b, prev = _q(np.stack([e[0], 2 * e[1] + 2 * e[2], e[3], e[4]]))
    cur_b, _ = _q(np.stack([e[0], 4 * e[1] + 4 * e[2], -e[3], e[5]]))
    assert oracle.drift(prev_b[:1], prev_b[:1]) == 0.0
    assert oracle.drift(prev_b[1:2], cur_b[1:2]) == pytest.approx(1.0, abs=1e-15)
    assert oracle.drift(prev_b[2:3], cur_b[2:3]) == pytest.approx(2.0, abs=1e-15)
    assert oracle.drift(prev_b[3:4], cur_b[3:4]) == pytest.approx(math.sqrt(2.0), abs=1e-15)
    assert oracle.drift(prev_b, cur_b) == pytest.approx((0 + 1 + 2 + math.sqrt(2)) / 4, abs=1e-15)


def test_stability_step_hand_trajectory():
    # t_i^*: the step at which a token's top prediction has been the same for
    # three consecutive decoded steps.  Gating off and a high fixed threshold
    # keep tokens masked unless their confidence is set above it.
    cfg = oracle.Config(B=1, P=4, T=8, n_blocks=2, theta_s=0.9,
                        flags=oracle.FIXED_THRESHOLD | oracle.DIAGNOSTICS)
    st = oracle.State(cfg)
    seq = [  # argmax per position at t = 0..4
        (5, 5, 5, 7),
        (5, 6, 6, 7),
        (5, 6, 5, 8),
        (5, 6, 6, 8),
        (5, 6, 5, 8),
    ]
    for t, idx in enumerate(seq):
        conf = np.full((1, 4), 0.01)
        if t == 1:
            conf[0, 3] = 0.95  # position 3 commits at t = 1, before it can be stable
        oracle.controller_step(st, 0, t, conf, np.array([idx], np.int32))
    assert list(st.stable[0, :4]) == [2, 3, -1, -1]
    assert list(st.run[0, :3]) == [5, 4, 1]
    # without the flag nothing is tracked
    plain = oracle.State(oracle.Config(B=1, P=4, T=8, n_blocks=2, flags=oracle.FIXED_THRESHOLD))
    for t, idx in enumerate(seq):
        oracle.controller_step(plain, 0, t, np.full((1, 4), 0.01), np.array([idx], np.int32))
    assert np.all(plain.stable == -1) and np.all(plain.run == 0)


def test_position_factor_printed():
    cfg = oracle.Config(P=64)
    for p, r in _rows("position_factors.txt"):
        assert oracle.pos_factor(cfg, int(p)) == float(r)
    off = oracle.Config(P=64, flags=oracle.GATING)
    assert oracle.pos_factor(off, 0) == 1.0 and oracle.pos_factor(off, 63) == 1.0
    q = oracle.Config(P=32, flags=oracle.POS_FACTOR | oracle.QUARTER_POS)
    assert [oracle.pos_factor(q, p) for p in (0, 7, 8, 15, 16, 23, 24, 31)] == \
        [0.8, 0.8, 0.9, 0.9, 1.05, 1.05, 1.1, 1.1]


def test_theta_token_clip():
    cfg = oracle.Config(T=32, P=64)
    # 0.90 * 1.10 = 0.99 is clipped to 0.98
    assert oracle.theta_token(cfg, 1, 0, 60) == pytest.approx(0.98, abs=1e-15)
    # 0.90 * 0.80 = 0.72 unclipped
    assert oracle.theta_token(cfg, 1, 0, 3) == pytest.approx(0.72, abs=1e-12)
    # block 4, last step: theta ~ 0.4017, times 0.80 -> 0.3213, unclipped
    assert oracle.theta_token(cfg, 4, 31, 0) == pytest.approx(0.401666 * 0.8, abs=1e-6)
    # a lower floor makes the 0.20 clip bite
    low = oracle.Config(T=32, P=64, theta_e1=0.2, theta_e_min=0.1)
    assert oracle.theta_token(low, 2, 31, 0) == pytest.approx(0.20, abs=1e-15)


def test_budget_table():
    cfg = oracle.Config(P=64)
    for p, s, bud in _rows("budget_table.txt"):
        assert oracle.budget(cfg, float(s), int(p)) == int(bud), (p, s)
    q = oracle.Config(P=32, flags=oracle.GATING | oracle.QUARTER_POS)
    assert oracle.budget(q, 0.9, 15) == 8 and oracle.budget(q, 0.9, 16) == 32
    assert oracle.budget(q, 0.9, 24) == 64


def test_low_yield_readings():
    cnt = oracle.Config()
    assert oracle.low_yield(cnt, 0) and oracle.low_yield(cnt, 1) and not oracle.low_yield(cnt, 2)
    frac = oracle.Config(eta_mode=1, eta_bar=0.015, n_blocks=8, P=32)   # L = 256, 1.5% = 3.84
    assert oracle.low_yield(frac, 3) and not oracle.low_yield(frac, 4)


# ------------------------------------------------------------- controller --

def _feed(cfg, seq):
    """Run controller steps on block 0 with per-step (conf[B,P], idx[B,P])."""
    st = oracle.State(cfg)
    for t, (c, i) in enumerate(seq):
        oracle.controller_step(st, 0, t, np.asarray(c, np.float64), np.asarray(i, np.int32))
        if np.all(st.exit_reason[:, 0] != oracle.RUNNING):
            break
    return st


def test_trajectory_G1_grinding_exit():
    # eta = 0, 0, 1, 0 -> ell = 1, 2, 3, 4 -> grinding at t = 3 (Box 7, K = 4).
    cfg = oracle.Config(B=1, P=4, T=10, n_blocks=1)
    idx = [[10, 11, 12, 13]]
    seq = [([[0.1, 0.1, 0.1, 0.1]], idx),
           ([[0.1, 0.1, 0.1, 0.1]], idx),
           ([[0.95, 0.1, 0.1, 0.1]], idx),
           ([[0.0, 0.41, 0.40, 0.2]], idx)]
    st = _feed(cfg, seq)
    assert st.exit_reason[0, 0] == oracle.EXIT_GRIND
    assert st.exit_step[0, 0] == 3
    assert st.ell[0] == 4
    # token 0 by threshold at t=2; token 1 forced (0.41 > 0.40); token 2 not (strict >)
    assert list(st.tok[0]) == [10, 11, -1, -1]
    assert list(st.cstep[0]) == [2, 3, -1, -1]
    assert st.unresolved[0, 0] == 2
    # all budgets 64 (s = 0.1 < 0.25)
    assert list(st.budget[0]) == [64] * 4


def test_trajectory_G2_counter_reset():
    # eta = 0, 2, 0, 0, 0, 0 -> ell = 1, 0, 1, 2, 3, 4 -> exit at t = 5.
    cfg = oracle.Config(B=1, P=6, T=10, n_blocks=1)
    idx = [list(range(6))]
    lo = [0.1] * 6
    seq = [([lo], idx), ([[0.99, 0.99] + [0.1] * 4], idx)] + [([lo], idx)] * 4
    ells = []
    st = oracle.State(cfg)
    for t, (c, i) in enumerate(seq):
        oracle.controller_step(st, 0, t, np.asarray(c), np.asarray(i, np.int32))
        ells.append(int(st.ell[0]))
    assert ells == [1, 0, 1, 2, 3, 4]
    assert st.exit_reason[0, 0] == oracle.EXIT_GRIND and st.exit_step[0, 0] == 5


@pytest.mark.parametrize("T,ending", [(8, oracle.EXIT_DONE), (3, oracle.EXIT_TMAX)])
def test_low_yield_counter_resets_at_each_block(T, ending):
    # Algorithm 1 sets ell <- 0 before each block's first step.  Block 0 commits
    # one token per step (eta = 1 < 1.5: ell = 1, 2, 3) and ends with ell = 3,
    # by DONE (P = 3, all committed at t = 2) or by T exhaustion (P = 4, T = 3).
    # Block 1's step zero commits nothing: with the reset ell = 1 and the block
    # runs on; without it ell = 4 = K and the block would exit by grinding at
    # t = 0.  The steps are fed to controller_step directly, so no caller-side
    # reset can stand in for the oracle's own.
    P = 3 if ending == oracle.EXIT_DONE else 4
    cfg = oracle.Config(B=1, P=P, T=T, n_blocks=2)
    idx = np.asarray([list(range(20, 20 + P))], np.int32)
    st = oracle.State(cfg)
    for t in range(3):
        c = np.full((1, P), 0.1)
        c[0, t] = 0.99                       # one commit per step (theta <= 0.90 * 1.0)
        oracle.controller_step(st, 0, t, c, idx)
        assert st.ell[0] == t + 1
    assert st.exit_reason[0, 0] == ending and st.exit_step[0, 0] == 2 and st.ell[0] == 3
    ells = []
    for t in range(min(T, 4)):
        oracle.controller_step(st, 1, t, np.full((1, P), 0.1), idx)
        ells.append(int(st.ell[0]))
        if t == 0:
            assert st.exit_reason[0, 1] == oracle.RUNNING, "ell carried over from block 0"
    assert ells == [1, 2, 3, 4][:len(ells)]
    if T >= 4:
        assert st.exit_reason[0, 1] == oracle.EXIT_GRIND and st.exit_step[0, 1] == 3
    # block 0's record is left as it was
    assert st.exit_reason[0, 0] == ending and list(st.tok[0, :3]) == [20, 21, 22]


def _budget_force_seq(P, T):
    # token 0: s = 0.6 at p = 0 -> B = 8; c stays 0.5 < theta.  Tokens 1..P-1
    # commit two per step (c = 0.99) so the low-yield counter stays at 0.
    seq = []
    for t in range(T):
        c = [0.5] + [0.0] * (P - 1)
        for j in (1 + 2 * t, 2 + 2 * t):
            if j < P:
                c[j] = 0.99
        c[0] = 0.6 if t == 0 else 0.5
        seq.append(([c], [list(range(100, 100 + P))]))
    return seq


def test_budget_force_commit_at_exactly_B():
    P, T = 22, 12
    cfg = oracle.Config(B=1, P=P, T=T, n_blocks=1)
    st = _feed(cfg, _budget_force_seq(P, T))
    assert st.budget[0, 0] == 8
    assert st.tok[0, 0] == 100 and st.cstep[0, 0] == 8
    # gating OFF: no budgets, token 0 is never committed by budget
    off = oracle.Config(B=1, P=P, T=T, n_blocks=1, flags=oracle.POS_FACTOR)
    st2 = _feed(off, _budget_force_seq(P, T))
    assert st2.tok[0, 0] == -1
    assert st2.exit_reason[0, 0] == oracle.EXIT_TMAX and st2.exit_step[0, 0] == T - 1


def test_done_exit_and_batch_independence():
    cfg = oracle.Config(B=2, P=3, T=8, n_blocks=2)
    idx = [[1, 2, 3], [4, 5, 6]]
    seq = [([[0.99, 0.99, 0.5], [0.99, 0.99, 0.99]], idx),
           ([[0.0, 0.0, 0.99], [0.0, 0.0, 0.0]], idx)]
    st = oracle.State(cfg)
    for t, (c, i) in enumerate(seq):
        oracle.controller_step(st, 0, t, np.asarray(c), np.asarray(i, np.int32))
    # sequence 1 finished at t = 0 (all three committed), sequence 0 at t = 1
    assert st.exit_reason[1, 0] == oracle.EXIT_DONE and st.exit_step[1, 0] == 0
    assert st.exit_reason[0, 0] == oracle.EXIT_DONE and st.exit_step[0, 0] == 1
    assert list(st.tok[0, :3]) == [1, 2, 3] and list(st.tok[1, :3]) == [4, 5, 6]
    # block 1 untouched
    assert np.all(st.tok[:, 3:] == -1)
    # an exited sequence ignores later steps
    oracle.controller_step(st, 0, 2, np.full((2, 3), 0.999), np.full((2, 3), 77, np.int32))
    assert list(st.tok[1, :3]) == [4, 5, 6]


def test_t_exhausted_and_flush():
    cfg = oracle.Config(B=1, P=2, T=3, n_blocks=1, flags=oracle.POS_FACTOR)
    idx = [[7, 8]]
    seq = [([[0.1, 0.2]], idx), ([[0.1, 0.2]], idx), ([[0.3, 0.95]], idx)]
    st = _feed(cfg, seq)
    assert st.exit_reason[0, 0] == oracle.EXIT_TMAX and st.exit_step[0, 0] == 2
    assert list(st.tok[0]) == [-1, 8] and st.unresolved[0, 0] == 1
    fl = oracle.Config(B=1, P=2, T=3, n_blocks=1, flags=oracle.POS_FACTOR | oracle.FLUSH_ON_EXIT)
    st2 = _feed(fl, seq)
    assert list(st2.tok[0]) == [7, 8] and st2.unresolved[0, 0] == 0
    assert list(st2.cstep[0]) == [2, 2]


def test_threshold_inclusive_and_position_factor_in_commit():
    # t = 0, theta_s = 0.9: p < 16 needs c >= 0.72 (inclusive), p in [16, 32) needs 0.81
    cfg = oracle.Config(B=1, P=32, T=32, n_blocks=1)
    c = np.full((1, 32), 0.1)
    th0 = oracle.theta_token(cfg, 1, 0, 0)     # 0.9 * 0.8 in double
    th17 = oracle.theta_token(cfg, 1, 0, 17)   # 0.9 * 0.9 in double
    assert th0 == pytest.approx(0.72, abs=1e-15) and th17 == pytest.approx(0.81, abs=1e-15)
    c[0, 0] = th0                        # exactly the threshold -> commits
    c[0, 1] = np.nextafter(th0, 0.0)     # one ulp below -> does not
    c[0, 16] = 0.80                      # below 0.81 -> does not
    c[0, 17] = th17                      # commits
    st = oracle.State(cfg)
    oracle.controller_step(st, 0, 0, c, np.arange(32, dtype=np.int32).reshape(1, 32))
    assert [st.tok[0, p] for p in (0, 1, 16, 17)] == [0, -1, -1, 17]
    assert st.eta[0] == 2


def _check_invariants(st: oracle.State, cfg: oracle.Config, history):
    """Invariants of Algorithm 1 over a finished trajectory."""
    gating = bool(cfg.flags & oracle.GATING)
    # committed tokens never change (history holds tok snapshots per step)
    for a, b in zip(history, history[1:]):
        done = a != -1
        assert np.all(b[done] == a[done])
    committed = st.tok != -1
    if gating:
        assert np.all(st.cstep[committed] <= st.budget[committed])
    for b in range(cfg.B):
        for blk in range(cfg.n_blocks):
            sl = slice(blk * cfg.P, (blk + 1) * cfg.P)
            cs = st.cstep[b, sl]
            if st.exit_step[b, blk] >= 0:
                assert np.all(cs[cs >= 0] <= st.exit_step[b, blk])
            assert st.unresolved[b, blk] == np.sum(st.tok[b, sl] == -1)


@pytest.mark.parametrize("mode", ["calibrated", "literal"])
def test_toy_trajectory_invariants(mode):
    wl = synth.WORKLOADS["toy"]
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w)
    hs = synth.HiddenStates(wl, W, mode)
    cfg = oracle.Config(B=wl.B, P=wl.P, T=wl.T, n_blocks=wl.n_blocks)
    history = []
    Ms = []
    etas = []

    def on_step(st, blk, t, out):
        history.append(st.tok.copy())
        Ms.append((blk, t, out["M"]))
        etas.append(int(st.eta.sum()))

    st = oracle.run_trajectory(cfg, W, hs, on_step=on_step)
    _check_invariants(st, cfg, history)
    # M_{t+1} = M_t - (tokens committed at t), within a block
    for k in range(len(Ms) - 1):
        (b0, t0, m0), (b1, t1, m1) = Ms[k], Ms[k + 1]
        if b0 == b1:
            before = np.sum(history[k - 1] != -1) if k > 0 else 0
            n_new = int(np.sum(history[k] != -1) - before)    # commits made at step k
            assert m1 == m0 - n_new
    if mode == "literal":
        # c ~ 1/V: every budget is 64 and every block exits by grinding at t = 3
        assert np.all(st.budget == 64)
        assert np.all(st.exit_reason == oracle.EXIT_GRIND) and np.all(st.exit_step == 3)
        assert np.all(st.tok == -1)


def test_theta_e_non_increasing_in_trajectory_configs():
    for nb in (4, 8, 16):
        cfg = oracle.Config(n_blocks=nb)
        vals = [oracle.theta_e(cfg, b) for b in range(1, nb + 1)]
        assert all(x >= y for x, y in zip(vals, vals[1:]))


# ------------------------------------------------- vocabulary-parallel head --

def _random_bf16(shape, scale, seed):
    rng = np.random.default_rng(seed)
    return bf16_from_float(rng.normal(0.0, scale, shape).astype(np.float32))


@pytest.mark.parametrize("cuts", [[], [500], [1, 999], [128, 333, 640], [7, 8, 9, 500, 990]])
def test_vocab_shards_merge_to_the_full_vocabulary(cuts):
    # Any partition of the vocabulary: the merged slice reductions equal Box 1
    # over the whole vocabulary (itself pinned by brute force above): the same
    # maximum and argmax, confidence and log-sum-exp to rounding.
    V, H, M = 1000, 64, 40
    W = _random_bf16((V, H), 0.05, 11)
    rows = _random_bf16((M, H), 1.0, 12)
    full = oracle.head_rows(W, rows)
    edges = [0] + cuts + [V]
    parts = [oracle.head_rows_shard(W[a:b], rows, a) for a, b in zip(edges[:-1], edges[1:])]
    got = oracle.merge_shards(parts)
    assert np.array_equal(got["idx"], full["idx"])
    assert np.array_equal(got["zmax"], full["zmax"])
    np.testing.assert_allclose(got["conf"], full["conf"], rtol=1e-12, atol=0)
    np.testing.assert_allclose(got["lse"], full["lse"], rtol=1e-12, atol=0)


def test_vocab_shards_tie_across_a_shard_boundary_keeps_the_lower_index():
    # Rows 37 and 537 of W are equal, and each hidden row points along them:
    # both logits are the maximum, in different shards.  The argmax is the
    # lower index (Box 1 with the lowest-index reading of ties), and c = 1/2
    # up to the other rows' tiny mass.
    V, H = 1000, 64
    W = _random_bf16((V, H), 0.02, 21)
    W[537] = W[37]
    w37 = np.frombuffer((W[37].astype(np.uint32) << 16).tobytes(), np.float32)
    rows = np.stack([bf16_from_float(w37 * 400.0 * (1 + 0.1 * k)) for k in range(3)])
    full = oracle.head_rows(W, rows)
    assert list(full["idx"]) == [37, 37, 37]
    parts = [oracle.head_rows_shard(W[:500], rows, 0), oracle.head_rows_shard(W[500:], rows, 500)]
    assert list(parts[1]["idx"]) == [537, 537, 537]
    got = oracle.merge_shards(parts)
    assert list(got["idx"]) == [37, 37, 37]
    np.testing.assert_allclose(got["conf"], full["conf"], rtol=1e-12)
    assert np.all(np.abs(got["conf"] - 0.5) < 1e-3)
    # the same split in the other order of the slices
    got2 = oracle.merge_shards(parts[::-1])
    assert list(got2["idx"]) == [37, 37, 37]


def test_vocab_shard_two_way_closed_form():
    # Two one-row slices: z = (a, b), so S over the whole vocabulary is
    # 1 + exp(-|a - b|) and c = sigma(|a - b|), whatever slice holds the max.
    H = 4
    for a, b in ((1.0, 0.0), (0.0, 2.5), (3.0, 3.0)):
        W = bf16_from_float(np.array([[a, 0, 0, 0], [b, 0, 0, 0]], np.float32))
        h = bf16_from_float(np.array([[1, 0, 0, 0]], np.float32))
        got = oracle.merge_shards([oracle.head_rows_shard(W[:1], h, 0),
                                   oracle.head_rows_shard(W[1:], h, 1)])
        assert got["conf"][0] == pytest.approx(1.0 / (1.0 + math.exp(-abs(a - b))), rel=1e-15)
        assert got["idx"][0] == (0 if a >= b else 1)
