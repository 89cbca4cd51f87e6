"""The parity harness's in-band substitution (no GPU): inside the tolerance
band the oracle must take the kernel's commit decisions, which the kernel
makes in fp32 (c >= theta_i, c > theta_fb, both thresholds rounded to fp32).
"""
import numpy as np

from tests.parity import kernel_side_value


def _kernel(c, theta, fb):
    c32 = np.float32(c)
    return bool(c32 >= np.float32(theta)), bool(c32 > np.float32(fb))


def _double(v, theta, fb):
    return bool(v >= theta), bool(v > fb)


def test_value_far_from_thresholds_is_the_kernels_own():
    c = np.float32(0.55)
    assert kernel_side_value(c, 0.77, 0.40) == float(c)


def test_one_ulp_below_the_double_threshold_commits_as_the_kernel_does():
    # theta_i whose fp32 rounding lies below it: an fp32 confidence equal to
    # that rounding commits on the kernel (c >= theta32) but not in fp64.
    theta = 0.7659490123456789
    t32 = np.float32(theta)
    assert float(t32) < theta
    v = kernel_side_value(t32, theta, 0.40)
    assert _double(v, theta, 0.40) == _kernel(t32, theta, 0.40) == (True, True)
    below = np.nextafter(t32, np.float32(0))
    v = kernel_side_value(below, theta, 0.40)
    assert _double(v, theta, 0.40) == _kernel(below, theta, 0.40) == (False, True)


def test_theta_above_its_fp32_rounding_and_strict_fallback_threshold():
    # theta_i rounded up in fp32, and theta_fb = 0.40 (rounded up in fp32:
    # an fp32 0.4 is not > theta_fb on the kernel, although it is in fp64).
    theta = 0.8000000000000001
    for c in (np.float32(theta), np.nextafter(np.float32(theta), np.float32(1)),
              np.float32(0.4), np.nextafter(np.float32(0.4), np.float32(1))):
        v = kernel_side_value(c, theta, 0.40)
        assert _double(v, theta, 0.40) == _kernel(c, theta, 0.40), c


def test_coinciding_thresholds():
    # theta_i = theta_fb = 0.4 (a clipped late threshold): c = fp32(0.4)
    # commits by theta_i (inclusive) and is not above theta_fb (strict).
    for c in (np.float32(0.4), np.nextafter(np.float32(0.4), np.float32(0)),
              np.nextafter(np.float32(0.4), np.float32(1))):
        v = kernel_side_value(c, 0.4, 0.4)
        assert _double(v, 0.4, 0.4) == _kernel(c, 0.4, 0.4), c


def test_random_values_near_thresholds():
    rng = np.random.default_rng(7)
    for _ in range(2000):
        theta = float(rng.uniform(0.3, 0.98))
        fb = 0.4
        c = np.float32(theta + rng.integers(-3, 4) * 6e-8)
        v = kernel_side_value(c, theta, fb)
        assert _double(v, theta, fb) == _kernel(c, theta, fb), (c, theta)


def _simulated_gpu_steps(B=6, P=16, T=8, seed=3):
    """States before and after each step of a synthetic trajectory, taken by
    the oracle's own controller on fp32-rounded confidences (standing in for
    the states a GPU step downloads), block 0 then block 1."""
    import oracle
    rng = np.random.default_rng(seed)
    cfg = oracle.Config(B=B, P=P, T=T, n_blocks=2)
    st = oracle.State(cfg)

    def dump(s):
        d = {f: getattr(s, f).copy() for f in oracle.State.FIELDS}
        d["conf"] = d["conf"].astype(np.float32)
        d["s0"] = d["s0"].astype(np.float32)
        d["m_hist"] = np.zeros((cfg.n_blocks, T), np.int32)
        return d

    pre = dump(st)
    steps = []
    for blk in range(2):
        for t in range(T):
            mk = st.masked(blk)
            conf = np.float32(rng.uniform(0.0, 1.0, (B, P))).astype(np.float64)
            idx = rng.integers(0, 1000, (B, P)).astype(np.int32)
            oracle.controller_step(st, blk, t, np.where(mk, conf, 0.0), np.where(mk, idx, -1))
            post = dump(st)
            post["m_hist"] = pre["m_hist"].copy()
            post["m_hist"][blk, t] = int(mk.sum())
            steps.append((blk, t, pre, post))
            pre = post
            if np.all(st.exit_reason[:, blk] != 0):
                break
    return cfg, steps


def test_controller_check_passes_on_a_consistent_step_and_catches_mistakes():
    from tests.parity import check_controller_step
    cfg, steps = _simulated_gpu_steps()
    assert len(steps) >= 4
    for blk, t, pre, post in steps:
        assert check_controller_step(cfg, pre, post, blk, t) == post["m_hist"][blk, t]
    # A committed token, a low-yield counter and M_t each changed in one
    # step's post state: the check must fail on each.
    blk, t, pre, post = next(s for s in steps if (s[3]["tok"] != s[2]["tok"]).any())
    for field, change in (("tok", lambda a: a.__setitem__(tuple(np.argwhere(
                              (post["tok"] != pre["tok"]))[0]), 999999)),
                          ("ell", lambda a: a.__setitem__(0, a[0] + 1)),
                          ("m_hist", lambda a: a.__setitem__((blk, t), a[blk, t] + 1))):
        bad = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in post.items()}
        change(bad[field])
        try:
            check_controller_step(cfg, pre, bad, blk, t)
        except AssertionError:
            continue
        raise AssertionError(f"a changed {field} was not caught")
