"""Python binding of the CAI-dLLM decoding-head library (``libcai.so``).

Argument marshalling only: every step of the decoding head and commit rule
runs in the library's sm_103a kernels (``csrc/``).  Function names follow the
C ABI in ``include/cai.h``.  Tensors are passed as PyTorch tensors (their
``data_ptr``) or raw integer pointers; streams as ``torch.cuda.Stream``, a raw
handle, or ``None`` for PyTorch's current stream.  A failing status raises
``CaiError`` carrying the status code.

There is no CPU fallback: the first call into the binding raises
``ImportError`` when the library is not built (``paper_2608_22646_gb300.build``).
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
# CAI_LIB selects another build of the library (e.g. libcai_debug.so).
LIB_PATH = os.environ.get("CAI_LIB") or os.path.join(_PKG, "libcai.so")

CAI_OK = 0
CAI_ERR_ARG = -1
CAI_ERR_SHAPE = -2
CAI_ERR_ORDER = -3
CAI_ERR_CUDA = -4
CAI_ERR_TIMEOUT = -5
CAI_ERR_DEVICE = -6
CAI_ERR_UNSUPPORTED = -7
CAI_ERR_NOMEM = -8

CAI_GATING = 1
CAI_POS_FACTOR = 2
CAI_FLUSH_ON_EXIT = 4
CAI_QUARTER_POS = 8
CAI_QUARTER_BLOCKS = 16
CAI_NO_BLOCK_SCHEDULE = 32
CAI_FIXED_THRESHOLD = 64
CAI_DIAGNOSTICS = 128

CAI_PRESET_LLADA = 0
CAI_PRESET_DREAM = 1

CAI_MASK_TOKEN = -1
CAI_RUNNING, CAI_EXIT_DONE, CAI_EXIT_GRIND, CAI_EXIT_TMAX = 0, 1, 2, 3

# Every symbol include/cai.h declares.
EXPORTS = ("cai_config_default", "cai_init", "cai_init_rmsnorm", "cai_first_step",
           "cai_denoise_step",
           "cai_block_advance", "cai_reset", "cai_poll", "cai_get_state", "cai_state_download",
           "cai_state_upload", "cai_read_tokens", "cai_profile", "cai_get_stats", "cai_free",
           "cai_strerror", "cai_test_fail_alloc_after", "cai_test_head_grid_limit",
           "cai_test_pair_plan", "cai_test_theta_table", "cai_test_wait_timeout",
           "cai_test_check_guards",
           "cai_head_rows_static", "cai_test_static_wait_timeout",
           "cai_init_vocab_shard", "cai_shard_rows", "cai_shard_head", "cai_shard_commit",
           "cai_device_error_bits")


class CaiError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        super().__init__(f"{what}: {status} ({cai_strerror(status)})")


class cai_config(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("P", ctypes.c_int32), ("H", ctypes.c_int32),
        ("V", ctypes.c_int32), ("T", ctypes.c_int32), ("n_blocks", ctypes.c_int32),
        ("theta_s", ctypes.c_double), ("theta_e1", ctypes.c_double),
        ("theta_e_step", ctypes.c_double), ("theta_e_min", ctypes.c_double),
        ("warmup_pct", ctypes.c_int32), ("K", ctypes.c_int32),
        ("theta_fb", ctypes.c_double), ("clip_lo", ctypes.c_double), ("clip_hi", ctypes.c_double),
        ("eta_bar", ctypes.c_double), ("eta_mode", ctypes.c_int32), ("flags", ctypes.c_uint32),
    ]


_STATE_FIELDS = ("tok", "conf", "s0", "budget", "cstep", "cand", "ell", "eta", "exit_reason",
                 "exit_step", "unresolved", "m_hist", "run", "stable", "drift")


class cai_state_view(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in _STATE_FIELDS]


class cai_host_state(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in _STATE_FIELDS] + [
        ("blk", ctypes.c_int32), ("t_next", ctypes.c_int32)]


class cai_stats(ctypes.Structure):
    _fields_ = [("steps", ctypes.c_int64), ("launches", ctypes.c_int64),
                ("head_launches", ctypes.c_int64), ("head_ms", ctypes.c_double),
                ("head_profiled", ctypes.c_int64), ("grid", ctypes.c_int32),
                ("stages", ctypes.c_int32), ("n_max", ctypes.c_int32),
                ("kernels_per_step", ctypes.c_int32), ("step_ms", ctypes.c_double),
                ("pair_grid", ctypes.c_int32), ("pair_swap_max_n", ctypes.c_int32),
                ("pair_stages", ctypes.c_int32), ("head_rows", ctypes.c_int32)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libcai.so is not built ({LIB_PATH}); run paper_2608_22646_gb300.build")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32 = ctypes.c_void_p, ctypes.c_int32
    sig = {
        "cai_config_default": (ctypes.c_int, [ctypes.POINTER(cai_config), i32, i32, i32, i32, i32, i32, i32]),
        "cai_init": (ctypes.c_int, [ctypes.POINTER(cai_config), vp, vp, ctypes.POINTER(vp)]),
        "cai_init_rmsnorm": (ctypes.c_int, [ctypes.POINTER(cai_config), vp, vp, ctypes.c_double, vp,
                                            ctypes.POINTER(vp)]),
        "cai_first_step": (ctypes.c_int, [vp, vp, vp]),
        "cai_denoise_step": (ctypes.c_int, [vp, vp, vp]),
        "cai_block_advance": (ctypes.c_int, [vp, vp]),
        "cai_reset": (ctypes.c_int, [vp, vp]),
        "cai_poll": (ctypes.c_int, [vp, i32, i32, ctypes.POINTER(i32)]),
        "cai_get_state": (ctypes.c_int, [vp, ctypes.POINTER(cai_state_view)]),
        "cai_state_download": (ctypes.c_int, [vp, ctypes.POINTER(cai_host_state)]),
        "cai_state_upload": (ctypes.c_int, [vp, ctypes.POINTER(cai_host_state)]),
        "cai_read_tokens": (ctypes.c_int, [vp, vp, vp]),
        "cai_profile": (ctypes.c_int, [vp, i32]),
        "cai_get_stats": (ctypes.c_int, [vp, ctypes.POINTER(cai_stats)]),
        "cai_device_error_bits": (ctypes.c_int, [vp, ctypes.POINTER(ctypes.c_uint32)]),
        "cai_free": (None, [vp]),
        "cai_strerror": (ctypes.c_char_p, [ctypes.c_int]),
        "cai_test_fail_alloc_after": (ctypes.c_int, [i32]),
        "cai_test_head_grid_limit": (ctypes.c_int, [i32]),
        "cai_test_pair_plan": (ctypes.c_int, [i32, i32, i32, ctypes.POINTER(i32)]),
        "cai_test_theta_table": (ctypes.c_int, [ctypes.POINTER(cai_config), i32, i32,
                                                ctypes.POINTER(ctypes.c_float)]),
        "cai_test_wait_timeout": (ctypes.c_int, [vp, vp]),
        "cai_test_check_guards": (ctypes.c_int, [vp, ctypes.POINTER(i32)]),
        "cai_head_rows_static": (ctypes.c_int, [vp, i32, i32, vp, i32, vp, vp, vp]),
        "cai_test_static_wait_timeout": (ctypes.c_int, []),
        "cai_init_vocab_shard": (ctypes.c_int, [ctypes.POINTER(cai_config), vp, i32, i32, vp,
                                                ctypes.POINTER(vp)]),
        "cai_shard_rows": (ctypes.c_int, [vp, ctypes.POINTER(i32)]),
        "cai_shard_head": (ctypes.c_int, [vp, vp, vp, vp]),
        "cai_shard_commit": (ctypes.c_int, [vp, vp, i32, vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = _load()
    return _lib


def _check(status: int, what: str):
    if status != CAI_OK:
        raise CaiError(status, what)


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    return x.data_ptr()


def _buf(x, what: str, dtype: str) -> int | None:
    """Address of a buffer the library reads or writes as a dense array of
    ``dtype`` ("bfloat16", "float32" or "int32"): a tensor or array of that
    element type with a contiguous layout, or a raw address (int).  A wrong
    element type or a strided view raises instead of being read as garbage."""
    if x is None or isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        # numpy has no bfloat16: such buffers travel as their uint16 bits
        want = {"bfloat16": np.uint16, "float32": np.float32, "int32": np.int32}[dtype]
        if x.dtype != want or not x.flags["C_CONTIGUOUS"]:
            raise ValueError(f"{what}: expected a C-contiguous {np.dtype(want)} array "
                             f"(got {x.dtype}, contiguous={x.flags['C_CONTIGUOUS']})")
        return x.ctypes.data
    if str(x.dtype) != f"torch.{dtype}" or not x.is_contiguous():
        raise ValueError(f"{what}: expected a contiguous torch.{dtype} tensor "
                         f"(got {x.dtype}, contiguous={x.is_contiguous()})")
    return x.data_ptr()


def _stream(s) -> int | None:
    if s is None:
        import torch
        if torch.cuda.is_available():
            return torch.cuda.current_stream().cuda_stream
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def cai_strerror(status: int) -> str:
    return lib().cai_strerror(status).decode()


def cai_config_default(preset: int, B: int, P: int, H: int, V: int, T: int, n_blocks: int) -> cai_config:
    c = cai_config()
    _check(lib().cai_config_default(ctypes.byref(c), preset, B, P, H, V, T, n_blocks),
           "cai_config_default")
    return c


class Ctx:
    """Owning handle of a ``cai_ctx*``; also keeps the sizes for the copies."""

    def __init__(self, handle: int, cfg: cai_config, W, norm_weight=None, norm_eps: float = 0.0):
        self.handle = handle
        self.cfg = cfg
        self._W = W  # read into the library's packed copies during cai_init
        self.norm_weight = norm_weight
        self.norm_eps = norm_eps

    @property
    def L(self) -> int:
        return self.cfg.n_blocks * self.cfg.P

    def __enter__(self) -> "Ctx":
        return self

    def __exit__(self, *exc) -> None:
        cai_free(self)


def cai_init(cfg: cai_config, W, stream=None) -> Ctx:
    h = ctypes.c_void_p()
    _check(lib().cai_init(ctypes.byref(cfg), _buf(W, "W", "bfloat16"), _stream(stream),
                          ctypes.byref(h)), "cai_init")
    return Ctx(h.value, cfg, W)


def cai_init_rmsnorm(cfg: cai_config, W, norm_weight, eps: float, stream=None) -> Ctx:
    """cai_init with the model's final RMSNorm (weight ``norm_weight`` [H] bf16,
    epsilon ``eps``) applied to every decoded row inside the head."""
    h = ctypes.c_void_p()
    _check(lib().cai_init_rmsnorm(ctypes.byref(cfg), _buf(W, "W", "bfloat16"),
                                  _buf(norm_weight, "norm_weight", "bfloat16"), float(eps),
                                  _stream(stream), ctypes.byref(h)), "cai_init_rmsnorm")
    return Ctx(h.value, cfg, W, norm_weight, float(eps))


def cai_init_vocab_shard(cfg: cai_config, W_shard, v0: int, stream=None) -> Ctx:
    """A shard context of the vocabulary-parallel head: ``W_shard`` [V_shard, H]
    holds the rows [v0, v0 + V_shard) of W; ``cfg.V`` is the whole vocabulary."""
    h = ctypes.c_void_p()
    _check(lib().cai_init_vocab_shard(ctypes.byref(cfg), _buf(W_shard, "W_shard", "bfloat16"),
                                      int(v0), int(W_shard.shape[0]), _stream(stream),
                                      ctypes.byref(h)), "cai_init_vocab_shard")
    return Ctx(h.value, cfg, W_shard)


def cai_shard_rows(ctx: Ctx) -> int:
    n = ctypes.c_int32(0)
    _check(lib().cai_shard_rows(ctx.handle, ctypes.byref(n)), "cai_shard_rows")
    return n.value


def cai_shard_head(ctx: Ctx, hidden, triples, stream=None) -> None:
    """This shard's triple of every masked row into ``triples``, a float32
    tensor [cai_shard_rows(ctx), 4] (the argmax travels as int32 bits)."""
    rows = cai_shard_rows(ctx)
    if not isinstance(triples, int) and tuple(triples.shape) != (rows, 4):
        raise ValueError(f"triples: expected shape ({rows}, 4), got {tuple(triples.shape)}")
    _check(lib().cai_shard_head(ctx.handle, _buf(hidden, "hidden", "bfloat16"),
                                _buf(triples, "triples", "float32"), _stream(stream)),
           "cai_shard_head")


def cai_shard_commit(ctx: Ctx, gathered, stream=None) -> None:
    """Merge every shard's triples, ``gathered`` float32 [n_shards, rows, 4],
    and apply the commit rule (ends the step)."""
    rows = cai_shard_rows(ctx)
    if gathered.ndim != 3 or tuple(gathered.shape[1:]) != (rows, 4):
        raise ValueError(f"gathered: expected shape (n_shards, {rows}, 4), "
                         f"got {tuple(gathered.shape)}")
    _check(lib().cai_shard_commit(ctx.handle, _buf(gathered, "gathered", "float32"),
                                  int(gathered.shape[0]), _stream(stream)), "cai_shard_commit")


def cai_first_step(ctx: Ctx, hidden, stream=None) -> None:
    _check(lib().cai_first_step(ctx.handle, _buf(hidden, "hidden", "bfloat16"), _stream(stream)),
           "cai_first_step")


def cai_denoise_step(ctx: Ctx, hidden, stream=None) -> None:
    _check(lib().cai_denoise_step(ctx.handle, _buf(hidden, "hidden", "bfloat16"), _stream(stream)),
           "cai_denoise_step")


def cai_block_advance(ctx: Ctx, stream=None) -> None:
    _check(lib().cai_block_advance(ctx.handle, _stream(stream)), "cai_block_advance")


def cai_reset(ctx: Ctx, stream=None) -> None:
    _check(lib().cai_reset(ctx.handle, _stream(stream)), "cai_reset")


def cai_poll(ctx: Ctx, lag: int = 0, timeout_ms: int = 10000) -> bool:
    done = ctypes.c_int32(0)
    _check(lib().cai_poll(ctx.handle, lag, timeout_ms, ctypes.byref(done)), "cai_poll")
    return bool(done.value)


def cai_get_state(ctx: Ctx) -> dict:
    v = cai_state_view()
    _check(lib().cai_get_state(ctx.handle, ctypes.byref(v)), "cai_get_state")
    return {n: getattr(v, n) for n in _STATE_FIELDS}


def _host_arrays(ctx: Ctx) -> dict:
    c = ctx.cfg
    B, L, nb = c.B, ctx.L, c.n_blocks
    return {
        "tok": np.zeros((B, L), np.int32), "conf": np.zeros((B, L), np.float32),
        "s0": np.zeros((B, L), np.float32), "budget": np.zeros((B, L), np.uint8),
        "cstep": np.zeros((B, L), np.int16), "cand": np.zeros((B, L), np.int32),
        "ell": np.zeros(B, np.int32), "eta": np.zeros(B, np.int32),
        "exit_reason": np.zeros((B, nb), np.int32), "exit_step": np.zeros((B, nb), np.int32),
        "unresolved": np.zeros((B, nb), np.int32), "m_hist": np.zeros((nb, c.T), np.int32),
        "run": np.zeros((B, L), np.uint8), "stable": np.zeros((B, L), np.int16),
        "drift": np.zeros((B, nb, c.T), np.float32),
    }


def cai_state_download(ctx: Ctx) -> dict:
    arrs = _host_arrays(ctx)
    hs = cai_host_state(**{n: arrs[n].ctypes.data for n in _STATE_FIELDS})
    _check(lib().cai_state_download(ctx.handle, ctypes.byref(hs)), "cai_state_download")
    arrs["blk"] = hs.blk
    arrs["t_next"] = hs.t_next
    return arrs


def cai_state_upload(ctx: Ctx, state: dict) -> None:
    ref = _host_arrays(ctx)
    keep = {}
    kw = {}
    for n in _STATE_FIELDS:
        if n in state and state[n] is not None:
            a = np.ascontiguousarray(state[n], dtype=ref[n].dtype).reshape(ref[n].shape)
            keep[n] = a
            kw[n] = a.ctypes.data
    hs = cai_host_state(**kw, blk=int(state["blk"]), t_next=int(state["t_next"]))
    _check(lib().cai_state_upload(ctx.handle, ctypes.byref(hs)), "cai_state_upload")


def cai_read_tokens(ctx: Ctx, host_tokens, stream=None) -> None:
    _check(lib().cai_read_tokens(ctx.handle, _buf(host_tokens, "host_tokens", "int32"),
                                 _stream(stream)), "cai_read_tokens")


def cai_profile(ctx: Ctx, enable: bool) -> None:
    _check(lib().cai_profile(ctx.handle, 1 if enable else 0), "cai_profile")


def cai_get_stats(ctx: Ctx) -> dict:
    s = cai_stats()
    _check(lib().cai_get_stats(ctx.handle, ctypes.byref(s)), "cai_get_stats")
    return {n: getattr(s, n) for n, _ in cai_stats._fields_}


DEVERR_NAMES = ("wait_empty", "wait_full", "wait_acc_full", "wait_acc_empty", "drain", "bad_row",
                "wait_epi", "bounds", "wait_rows")


def cai_device_error_bits(ctx: Ctx) -> int:
    """The context's device error word (bit k: DEVERR_NAMES[k]); works on a
    context that returned CAI_ERR_DEVICE."""
    v = ctypes.c_uint32(0)
    _check(lib().cai_device_error_bits(ctx.handle, ctypes.byref(v)), "cai_device_error_bits")
    return int(v.value)


def cai_free(ctx: Ctx) -> None:
    if ctx.handle:
        lib().cai_free(ctx.handle)
        ctx.handle = 0


def cai_test_fail_alloc_after(n: int) -> None:
    _check(lib().cai_test_fail_alloc_after(n), "cai_test_fail_alloc_after")


def cai_test_wait_timeout(ctx: Ctx, stream=None) -> None:
    _check(lib().cai_test_wait_timeout(ctx.handle, _stream(stream)), "cai_test_wait_timeout")


def cai_test_pair_plan(M: int, n_pairs: int, swap_max_n: int) -> dict:
    out = (ctypes.c_int32 * 4)()
    _check(lib().cai_test_pair_plan(M, n_pairs, swap_max_n, out), "cai_test_pair_plan")
    return {"swapped": bool(out[0]), "row_tiles": out[1], "tile_rows": out[2],
            "partials_per_row": out[3]}


def cai_test_theta_table(cfg: cai_config, blk: int, t: int) -> np.ndarray:
    """theta_i(t) of every position of block ``blk`` at local step ``t``, as
    the step's commit rule receives it (fp32)."""
    out = np.zeros(cfg.P, np.float32)
    _check(lib().cai_test_theta_table(ctypes.byref(cfg), blk, t,
                                      out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))),
           "cai_test_theta_table")
    return out


def cai_test_head_grid_limit(n: int) -> None:
    _check(lib().cai_test_head_grid_limit(n), "cai_test_head_grid_limit")


def cai_test_check_guards(ctx: Ctx) -> int:
    """Number of the context's device buffers written past their end."""
    n = ctypes.c_int32(0)
    _check(lib().cai_test_check_guards(ctx.handle, ctypes.byref(n)), "cai_test_check_guards")
    return n.value


def cai_head_rows_static(W, rows, conf, argmax, stream=None) -> None:
    """Confidence and argmax of every row of ``rows`` [M, H] against ``W`` [V, H]
    into the device arrays ``conf`` (float32 [M]) and ``argmax`` (int32 [M]),
    allocating nothing (see include/cai.h)."""
    V, H = W.shape
    M = rows.shape[0]
    _check(lib().cai_head_rows_static(_buf(W, "W", "bfloat16"), V, H, _buf(rows, "rows", "bfloat16"),
                                      M, _buf(conf, "conf", "float32"),
                                      _buf(argmax, "argmax", "int32"), _stream(stream)),
           "cai_head_rows_static")


def cai_test_static_wait_timeout() -> None:
    """Make the next cai_head_rows_static call record a failed bounded wait."""
    _check(lib().cai_test_static_wait_timeout(), "cai_test_static_wait_timeout")


def config_from_dict(d: dict) -> cai_config:
    c = cai_config()
    for k, v in d.items():
        setattr(c, k, v)
    return c
