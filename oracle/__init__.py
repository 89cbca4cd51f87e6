"""CAI-dLLM oracle: TEST INFRASTRUCTURE ONLY.

Python marshalling around ``cai_oracle.c``, the plain fp64 CPU statement of the
decoding head (Box 1) and the confidence-aware controller (Boxes 2-7,
Algorithm 1) of arXiv 2608.22646, plus the block loop of Algorithm 1 run over a
batch in lockstep.

Only ``tests/``, ``__graft_entry__.smoke()``, the CPU-baseline leg and the
reference arm of ``bench.py``, and ``calibrate_synth.py`` beside this file may
import this package.  It shares no code with the CUDA path and
never imports it.  bf16 tensors cross this boundary as ``uint16`` bit patterns.

Parity status of each function (what pins it, beyond itself) is listed in
``tests/test_oracle_pins.py``; every function here is pinned.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cai_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

GATING = 1
POS_FACTOR = 2
FLUSH_ON_EXIT = 4
QUARTER_POS = 8
QUARTER_BLOCKS = 16
NO_BLOCK_SCHEDULE = 32   # Box 3 alone: theta_e1 in every block ("APD" ablation row)
FIXED_THRESHOLD = 64     # fixed-threshold rule (Fast-dLLM): theta = theta_s always
DIAGNOSTICS = 128        # stability step t_i^* and drift D^(t) (Section 2.1)

MASK = -1
RUNNING, EXIT_DONE, EXIT_GRIND, EXIT_TMAX = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math: IEEE double semantics)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-pthread", "-fno-fast-math",
             "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


class _Cfg(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("P", ctypes.c_int32), ("T", ctypes.c_int32),
        ("n_blocks", ctypes.c_int32),
        ("theta_s", ctypes.c_double), ("theta_e1", ctypes.c_double),
        ("theta_e_step", ctypes.c_double), ("theta_e_min", ctypes.c_double),
        ("warmup_pct", ctypes.c_int32), ("K", ctypes.c_int32),
        ("theta_fb", ctypes.c_double), ("clip_lo", ctypes.c_double),
        ("clip_hi", ctypes.c_double), ("eta_bar", ctypes.c_double),
        ("eta_mode", ctypes.c_int32), ("flags", ctypes.c_uint32),
    ]


class _State(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "tok", "conf", "s0", "budget", "cstep", "cand", "ell", "eta",
        "exit_reason", "exit_step", "unresolved", "run", "stable")]


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        d, i32, u16p = ctypes.c_double, ctypes.c_int32, ctypes.c_void_p
        cfgp = ctypes.POINTER(_Cfg)
        _lib.cai_o_bf16_to_double.restype = d
        _lib.cai_o_bf16_to_double.argtypes = [ctypes.c_uint16]
        _lib.cai_o_head_rows.restype = i32
        _lib.cai_o_head_rows.argtypes = [u16p, i32, i32, u16p, i32, i32,
                                         u16p, u16p, u16p, u16p, u16p]
        _lib.cai_o_head_rows_norm.restype = i32
        _lib.cai_o_head_rows_norm.argtypes = [u16p, i32, i32, u16p, i32, u16p, d, i32,
                                              u16p, u16p, u16p, u16p, u16p]
        _lib.cai_o_drift.restype = d
        _lib.cai_o_drift.argtypes = [u16p, u16p, i32, i32]
        _lib.cai_o_softmax_row.restype = i32
        _lib.cai_o_softmax_row.argtypes = [u16p, i32, i32, u16p, u16p, u16p]
        for name in ("cai_o_theta_e",):
            getattr(_lib, name).restype = d
            getattr(_lib, name).argtypes = [cfgp, i32]
        _lib.cai_o_theta_block.restype = d
        _lib.cai_o_theta_block.argtypes = [cfgp, i32, i32]
        _lib.cai_o_pos_factor.restype = d
        _lib.cai_o_pos_factor.argtypes = [cfgp, i32]
        _lib.cai_o_theta_token.restype = d
        _lib.cai_o_theta_token.argtypes = [cfgp, i32, i32, i32]
        _lib.cai_o_budget.restype = i32
        _lib.cai_o_budget.argtypes = [cfgp, d, i32]
        _lib.cai_o_low_yield.restype = i32
        _lib.cai_o_low_yield.argtypes = [cfgp, i32]
        _lib.cai_o_controller_step.restype = None
        _lib.cai_o_controller_step.argtypes = [cfgp, ctypes.POINTER(_State), i32, i32, u16p, u16p]
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


@dataclass
class Config:
    """Controller hyperparameters.  Defaults are the paper's (Boxes 3-7,
    Section 5 "Decoding settings") with gating ON, position factors ON."""
    B: int = 1
    P: int = 32
    T: int = 32
    n_blocks: int = 8
    theta_s: float = 0.90
    theta_e1: float = 0.70
    theta_e_step: float = 0.10
    theta_e_min: float = 0.40
    warmup_pct: int = 15
    K: int = 4
    theta_fb: float = 0.40
    clip_lo: float = 0.20
    clip_hi: float = 0.98
    eta_bar: float = 1.5
    eta_mode: int = 0
    flags: int = GATING | POS_FACTOR

    def c(self) -> _Cfg:
        return _Cfg(self.B, self.P, self.T, self.n_blocks, self.theta_s, self.theta_e1,
                    self.theta_e_step, self.theta_e_min, self.warmup_pct, self.K, self.theta_fb,
                    self.clip_lo, self.clip_hi, self.eta_bar, self.eta_mode, self.flags)


# ------------------------------------------------------------------ head --

def bf16_bits(x) -> np.ndarray:
    """Accept a torch bf16 tensor or a uint16 ndarray; return uint16 bits."""
    if isinstance(x, np.ndarray):
        assert x.dtype == np.uint16
        return np.ascontiguousarray(x)
    import torch
    assert x.dtype == torch.bfloat16
    return np.ascontiguousarray(x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))


def head_rows(W, rows, n_threads: int | None = None, norm_weight=None, eps: float = 0.0) -> dict:
    """Box 1 for every row of ``rows`` [M, H] against ``W`` [V, H] (bf16).
    With ``norm_weight`` g [H] (bf16), each row h is first put through the
    model's final RMSNorm, g * h / sqrt(mean(h^2) + eps), in fp64.

    Returns conf (c = max_v p), idx (argmax, lowest index on ties), zmax,
    lse (log-sum-exp) and gap (top-1 minus top-2 logit), all fp64/int32."""
    Wb, Rb = bf16_bits(W), bf16_bits(rows)
    V, H = Wb.shape
    Rb = Rb.reshape(-1, H)
    M = Rb.shape[0]
    out = {k: np.zeros(M, np.float64) for k in ("conf", "zmax", "lse", "gap")}
    out["idx"] = np.zeros(M, np.int32)
    if n_threads is None:
        n_threads = os.cpu_count() or 1
    gb = None
    if norm_weight is not None:
        gb = bf16_bits(norm_weight).reshape(-1)
        assert gb.shape[0] == H
    rc = lib().cai_o_head_rows_norm(_ptr(Wb), V, H, _ptr(Rb), M,
                                    None if gb is None else _ptr(gb), float(eps), n_threads,
                                    _ptr(out["conf"]), _ptr(out["idx"]), _ptr(out["zmax"]),
                                    _ptr(out["lse"]), _ptr(out["gap"]))
    if rc != 0:
        raise RuntimeError(f"oracle head failed: {rc}")
    return out


def head_rows_shard(W_shard, rows, v0: int, n_threads: int | None = None) -> dict:
    """Box 1's three reductions over one slice of the vocabulary, the rows
    [v0, v0 + V_shard) of W held as ``W_shard`` [V_shard, H] (bf16): per row
    m = max_v z_v over the slice, S = sum over the slice of exp(z_v - m), and
    idx = the lowest (global) index v of the slice with z_v = m.  The
    vocabulary-parallel head computes these on every shard and merges them
    (``merge_shards``)."""
    h = head_rows(W_shard, rows, n_threads)
    return {"m": h["zmax"], "S": 1.0 / h["conf"], "idx": h["idx"].astype(np.int64) + int(v0)}


def merge_shards(parts) -> dict:
    """Box 1 over the whole vocabulary from the reductions of the slices of
    any partition of it (``head_rows_shard`` of each): m = max_k m_k,
    S = sum_k S_k exp(m_k - m), the argmax the lowest idx_k among the slices
    whose m_k equals m (ties keep the lowest index), c = 1 / S."""
    m = np.max(np.stack([p["m"] for p in parts]), axis=0)
    S = np.sum(np.stack([p["S"] * np.exp(p["m"] - m) for p in parts]), axis=0)
    big = np.iinfo(np.int64).max
    idx = np.min(np.stack([np.where(p["m"] == m, p["idx"], big) for p in parts]), axis=0)
    return {"conf": 1.0 / S, "idx": idx.astype(np.int32), "zmax": m, "lse": m + np.log(S)}


def softmax_row(W, h):
    """Logits and full probability vector of one row (Box 1)."""
    Wb, hb = bf16_bits(W), bf16_bits(h).reshape(-1)
    V, H = Wb.shape
    z = np.zeros(V, np.float64)
    p = np.zeros(V, np.float64)
    idx = lib().cai_o_softmax_row(_ptr(Wb), V, H, _ptr(hb), _ptr(z), _ptr(p))
    return z, p, idx


# ------------------------------------------------------------ scalar rules --

def theta_e(cfg: Config, b: int) -> float:
    c = cfg.c()
    return lib().cai_o_theta_e(ctypes.byref(c), b)


def theta_block(cfg: Config, b: int, t: int) -> float:
    c = cfg.c()
    return lib().cai_o_theta_block(ctypes.byref(c), b, t)


def pos_factor(cfg: Config, p: int) -> float:
    c = cfg.c()
    return lib().cai_o_pos_factor(ctypes.byref(c), p)


def theta_token(cfg: Config, b: int, t: int, p: int) -> float:
    c = cfg.c()
    return lib().cai_o_theta_token(ctypes.byref(c), b, t, p)


def budget(cfg: Config, s: float, p: int) -> int:
    c = cfg.c()
    return lib().cai_o_budget(ctypes.byref(c), s, p)


def low_yield(cfg: Config, eta: int) -> bool:
    c = cfg.c()
    return bool(lib().cai_o_low_yield(ctypes.byref(c), eta))


# -------------------------------------------------------------- controller --

@dataclass
class State:
    """Controller state of a whole generation: per-token arrays are [B, L]
    with L = n_blocks * P; per-block arrays are [B, n_blocks]."""
    cfg: Config
    tok: np.ndarray = field(init=False)
    conf: np.ndarray = field(init=False)
    s0: np.ndarray = field(init=False)
    budget: np.ndarray = field(init=False)
    cstep: np.ndarray = field(init=False)
    cand: np.ndarray = field(init=False)
    ell: np.ndarray = field(init=False)
    eta: np.ndarray = field(init=False)
    exit_reason: np.ndarray = field(init=False)
    exit_step: np.ndarray = field(init=False)
    unresolved: np.ndarray = field(init=False)
    run: np.ndarray = field(init=False)
    stable: np.ndarray = field(init=False)

    def __post_init__(self):
        B, L, nb = self.cfg.B, self.cfg.n_blocks * self.cfg.P, self.cfg.n_blocks
        self.tok = np.full((B, L), MASK, np.int32)
        self.conf = np.zeros((B, L), np.float64)
        self.s0 = np.zeros((B, L), np.float64)
        self.budget = np.zeros((B, L), np.int32)
        self.cstep = np.full((B, L), -1, np.int32)
        self.cand = np.full((B, L), -1, np.int32)
        self.ell = np.zeros(B, np.int32)
        self.eta = np.zeros(B, np.int32)
        self.exit_reason = np.zeros((B, nb), np.int32)
        self.exit_step = np.full((B, nb), -1, np.int32)
        self.unresolved = np.zeros((B, nb), np.int32)
        self.run = np.zeros((B, L), np.int32)
        self.stable = np.full((B, L), -1, np.int32)

    FIELDS = ("tok", "conf", "s0", "budget", "cstep", "cand", "ell", "eta",
              "exit_reason", "exit_step", "unresolved", "run", "stable")

    def copy(self) -> "State":
        s = State(self.cfg)
        for f in self.FIELDS:
            setattr(s, f, getattr(self, f).copy())
        return s

    def _c(self) -> _State:
        return _State(*[getattr(self, f).ctypes.data for f in self.FIELDS])

    def masked(self, blk: int) -> np.ndarray:
        """[B, P] bool: still-masked tokens of running sequences in block blk."""
        P = self.cfg.P
        m = self.tok[:, blk * P:(blk + 1) * P] == MASK
        running = self.exit_reason[:, blk] == RUNNING
        return m & running[:, None]


def drift(h_prev, h_cur) -> float:
    """Eq. relative_drift for one sequence: mean over positions of
    ||h_cur - h_prev|| / ||h_prev||; rows [P, H] bf16."""
    a, b = bf16_bits(h_prev), bf16_bits(h_cur)
    H = a.shape[-1]
    a, b = a.reshape(-1, H), b.reshape(-1, H)
    assert a.shape == b.shape
    return float(lib().cai_o_drift(_ptr(a), _ptr(b), a.shape[0], H))


def controller_step(st: State, blk: int, t: int, conf_bp: np.ndarray, idx_bp: np.ndarray):
    """Algorithm 1, commit loop through the exit checks, for all sequences."""
    cfg = st.cfg
    conf_bp = np.ascontiguousarray(conf_bp, np.float64).reshape(cfg.B, cfg.P)
    idx_bp = np.ascontiguousarray(idx_bp, np.int32).reshape(cfg.B, cfg.P)
    c = cfg.c()
    cs = st._c()
    lib().cai_o_controller_step(ctypes.byref(c), ctypes.byref(cs), blk, t, _ptr(conf_bp), _ptr(idx_bp))


def step(st: State, W, hidden_bph, blk: int, t: int, n_threads: int | None = None,
         norm_weight=None, eps: float = 0.0) -> dict:
    """One denoising step: the head (after the final RMSNorm when
    ``norm_weight`` is given) on every masked row of a running sequence (rows
    taken in (b, p) order), then the controller.  Returns the head outputs
    scattered to [B, P] (NaN / -1 where not computed) and M_t."""
    cfg = st.cfg
    hb = bf16_bits(hidden_bph).reshape(cfg.B, cfg.P, -1)
    mk = st.masked(blk)
    rows = hb[mk]
    M = rows.shape[0]
    conf = np.full((cfg.B, cfg.P), np.nan)
    idx = np.full((cfg.B, cfg.P), -1, np.int32)
    gap = np.full((cfg.B, cfg.P), np.nan)
    if M:
        h = head_rows(W, np.ascontiguousarray(rows), n_threads, norm_weight, eps)
        conf[mk], idx[mk], gap[mk] = h["conf"], h["idx"], h["gap"]
    controller_step(st, blk, t, np.nan_to_num(conf), idx)
    return {"conf": conf, "idx": idx, "gap": gap, "M": M, "masked": mk}


def run_trajectory(cfg: Config, W, hidden_fn, n_threads: int | None = None, on_step=None) -> State:
    """Algorithm 1 over all blocks, batch in lockstep.

    ``hidden_fn(blk, t)`` returns the [B, P, H] bf16 hidden states of block
    ``blk`` at local step ``t``.  ``on_step(st, blk, t, out)`` is called after
    every step (tests use it to compare or re-synchronise state)."""
    st = State(cfg)
    for blk in range(cfg.n_blocks):
        # (the controller itself sets ell <- 0 at each block's step zero)
        for t in range(cfg.T):
            out = step(st, W, hidden_fn(blk, t), blk, t, n_threads)
            if on_step is not None:
                on_step(st, blk, t, out)
            if np.all(st.exit_reason[:, blk] != RUNNING):
                break
    return st
