"""The C ABI on a machine without a GPU: the library loads, exports exactly
what include/cai.h declares, its structs have the header's layout, and
argument / shape validation answers before any CUDA call."""
import ctypes
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

import paper_2608_22646_gb300 as cai

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cai.h")


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_22646_gb300 import build
    build.build()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(cai_[a-z0-9_]+)\s*\(", src)))


def test_exports_match_header():
    names = _declared()
    assert names == sorted(cai.EXPORTS), (names, sorted(cai.EXPORTS))
    lib = cai.lib()
    for n in names:
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", cai.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (cai_[a-z0-9_]+)$", out, flags=re.M))
    assert set(names) <= exported


def _c_layout():
    """sizeof/offsetof of the ABI structs as a C compiler sees the header."""
    prog = r'''
#include <stddef.h>
#include <stdio.h>
#include "cai.h"
#define F(T, f) printf(#T "." #f " %zu\n", offsetof(T, f));
int main(void) {
  printf("cai_config %zu\ncai_state_view %zu\ncai_host_state %zu\ncai_stats %zu\n",
         sizeof(cai_config), sizeof(cai_state_view), sizeof(cai_host_state), sizeof(cai_stats));
  F(cai_config, theta_s) F(cai_config, warmup_pct) F(cai_config, theta_fb) F(cai_config, eta_bar)
  F(cai_config, eta_mode) F(cai_config, flags)
  F(cai_host_state, m_hist) F(cai_host_state, blk) F(cai_host_state, t_next)
  F(cai_stats, head_ms) F(cai_stats, grid) F(cai_stats, n_max)
  return 0;
}
'''
    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "l.c")
        open(c, "w").write(prog)
        exe = os.path.join(d, "l")
        subprocess.check_call(["gcc", "-std=c99", "-I", os.path.dirname(HEADER), c, "-o", exe])
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout
    return dict(line.rsplit(" ", 1) for line in out.strip().splitlines())


def test_struct_layout_matches_binding():
    lay = {k: int(v) for k, v in _c_layout().items()}
    assert lay["cai_config"] == ctypes.sizeof(cai.cai_config)
    assert lay["cai_state_view"] == ctypes.sizeof(cai.cai_state_view)
    assert lay["cai_host_state"] == ctypes.sizeof(cai.cai_host_state)
    assert lay["cai_stats"] == ctypes.sizeof(cai.cai_stats)
    for key, v in lay.items():
        if "." in key:
            s, f = key.split(".")
            assert getattr(getattr(cai, s), f).offset == v, key


def test_config_default_values():
    c = cai.cai_config_default(cai.CAI_PRESET_LLADA, 1, 32, 4096, 126464, 32, 8)
    assert (c.theta_s, c.theta_e1, c.theta_e_step, c.theta_e_min) == (0.9, 0.7, 0.1, 0.4)
    assert (c.warmup_pct, c.K, c.theta_fb, c.clip_lo, c.clip_hi, c.eta_bar) == \
        (15, 4, 0.4, 0.2, 0.98, 1.5)
    assert c.flags == cai.CAI_GATING | cai.CAI_POS_FACTOR
    d = cai.cai_config_default(cai.CAI_PRESET_DREAM, 1, 32, 3584, 152064, 32, 8)
    assert d.flags == cai.CAI_POS_FACTOR
    with pytest.raises(cai.CaiError) as e:
        cai.cai_config_default(7, 1, 1, 64, 64, 1, 1)
    assert e.value.status == cai.CAI_ERR_ARG


@pytest.mark.parametrize("field,value,status", [
    ("H", 100, cai.CAI_ERR_SHAPE),      # H % 64 != 0
    ("P", 300, cai.CAI_ERR_SHAPE),      # P > 256
    ("V", 32, cai.CAI_ERR_SHAPE),       # V < 64
    ("B", 0, cai.CAI_ERR_SHAPE),
    ("T", 0, cai.CAI_ERR_SHAPE),
    ("n_blocks", 40000, cai.CAI_ERR_SHAPE),
    ("K", 0, cai.CAI_ERR_ARG),
    ("eta_mode", 2, cai.CAI_ERR_ARG),
    ("flags", 1 << 8, cai.CAI_ERR_ARG),
])
def test_init_validates_before_any_cuda_call(field, value, status):
    c = cai.cai_config_default(0, 1, 16, 256, 4096, 8, 4)
    setattr(c, field, value)
    w = (ctypes.c_uint16 * 16)()
    h = ctypes.c_void_p()
    assert cai.lib().cai_init(ctypes.byref(c), ctypes.addressof(w), None, ctypes.byref(h)) == status
    assert not h.value


def test_null_and_status_strings():
    lib = cai.lib()
    h = ctypes.c_void_p()
    assert lib.cai_init(None, None, None, ctypes.byref(h)) == cai.CAI_ERR_ARG
    for fn in ("cai_first_step", "cai_denoise_step"):
        assert getattr(lib, fn)(None, None, None) == cai.CAI_ERR_ARG
    assert lib.cai_block_advance(None, None) == cai.CAI_ERR_ARG
    lib.cai_free(None)
    for s in range(-8, 1):
        assert cai.cai_strerror(s) != "unknown status"
    assert cai.cai_strerror(-99) == "unknown status"
    assert lib.cai_test_fail_alloc_after(-1) == cai.CAI_ERR_ARG
    assert lib.cai_test_head_grid_limit(-1) == cai.CAI_ERR_ARG
    assert lib.cai_test_wait_timeout(None, None) == cai.CAI_ERR_ARG


def test_no_device_is_a_status_not_a_crash():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    c = cai.cai_config_default(0, 1, 16, 256, 4096, 8, 4)
    w = (ctypes.c_uint16 * (4096 * 256))()
    h = ctypes.c_void_p()
    r = cai.lib().cai_init(ctypes.byref(c), ctypes.addressof(w), None, ctypes.byref(h))
    assert r in (cai.CAI_ERR_CUDA, cai.CAI_ERR_UNSUPPORTED) and not h.value


@pytest.mark.parametrize("n_pairs", [76, 74, 3, 1])
def test_pair_plan_covers_rows_with_bounded_padding(n_pairs):
    # The pair LM head's per-step plan (host logic, no device): row tiles of
    # at most 256 rows cover M; swapped tiles are equal, a multiple of 32
    # wide, and pad fewer than 32 rows each; a step is swapped exactly when
    # its tile would be at most swap_max_n wide; one partial per pair (and
    # CTA when swapped) exactly when the row-tile count divides the pairs.
    for max_n in (0, 32, 192, 256):
        for M in range(1, 2049):
            pl = cai.cai_test_pair_plan(M, n_pairs, max_n)
            n_rt = -(-M // 256)
            assert pl["row_tiles"] == n_rt
            width = -(-(-(-M // n_rt)) // 32) * 32
            assert 32 <= width <= 256 and n_rt * width >= M
            assert n_rt * width - M < 32 * n_rt
            assert pl["swapped"] == (max_n >= 32 and width <= max_n), (M, max_n)
            assert pl["tile_rows"] == (width if pl["swapped"] else 256)
            if pl["swapped"]:
                assert pl["tile_rows"] * n_rt - M < 32 * n_rt
            want = 0 if n_pairs % n_rt else (2 if pl["swapped"] else 1) * (n_pairs // n_rt)
            assert pl["partials_per_row"] == want
    lib = cai.lib()
    out = (ctypes.c_int32 * 4)()
    assert lib.cai_test_pair_plan(0, 76, 192, out) == cai.CAI_ERR_ARG
    assert lib.cai_test_pair_plan(5, 0, 192, out) == cai.CAI_ERR_ARG
    assert lib.cai_test_pair_plan(5, 76, -1, out) == cai.CAI_ERR_ARG
    assert lib.cai_test_pair_plan(5, 76, 192, None) == cai.CAI_ERR_ARG


def test_bench_reference_arm_json_line():
    # The reference arm (the oracle on the host cores) needs no GPU: one JSON
    # line with the contract's fields, its own cpu_baseline and e2e.
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "toy",
                          "--steps", "2", "--warmup", "3"], cwd=root, capture_output=True,
                         text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["unit"] == "positions/s"
    assert line["higher_is_better"] is True and line["steps"] == 2 and line["warmup"] == 3
    for k in ("metric", "n_gpus", "ms_per_step", "scaling", "dtype", "data", "config"):
        assert k in line, k
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]


def test_binding_rejects_wrong_element_types_and_strided_views():
    # The library reads W and the hidden states as dense bf16, the tokens as
    # int32: the binding raises on anything else instead of passing a pointer.
    import torch
    from paper_2608_22646_gb300 import _buf
    w = torch.zeros((8, 64), dtype=torch.bfloat16)
    assert _buf(w, "W", "bfloat16") == w.data_ptr()
    assert _buf(1234, "W", "bfloat16") == 1234 and _buf(None, "W", "bfloat16") is None
    for bad in (w.float(), w.half(), w.t(), w[:, ::2]):
        with pytest.raises(ValueError):
            _buf(bad, "W", "bfloat16")
    bits = np.zeros((8, 64), np.uint16)
    assert _buf(bits, "W", "bfloat16") == bits.ctypes.data
    with pytest.raises(ValueError):
        _buf(bits[:, ::2], "W", "bfloat16")
    with pytest.raises(ValueError):
        _buf(np.zeros(8, np.float32), "W", "bfloat16")
    tok = torch.zeros((2, 5), dtype=torch.int32)
    assert _buf(tok, "host_tokens", "int32") == tok.data_ptr()
    with pytest.raises(ValueError):
        _buf(tok.long(), "host_tokens", "int32")


def test_context_handle_frees_on_exit():
    c = cai.cai_config_default(0, 1, 16, 256, 4096, 8, 4)
    with cai.Ctx(0, c, None) as ctx:     # a null handle: nothing to free
        assert ctx.L == 64
    assert ctx.handle == 0


def _golden(name):
    out = []
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                out.append(line.split())
    return out


def test_theta_table_matches_golden_schedule_and_position_factors():
    # The product's host-side threshold table (what the commit rule receives)
    # against the hand-worked Box 3-4 schedule and the printed Box 6 factors.
    for T, b, t, th in _golden("theta_schedule.txt"):
        T, b, t, th = int(T), int(b), int(t), float(th)
        c = cai.cai_config_default(0, 1, 16, 256, 4096, T, max(4, b))
        c.flags = 0                                   # no position factors
        tab = cai.cai_test_theta_table(c, b - 1, t)
        assert abs(float(tab[0]) - th) <= 6e-7, (T, b, t, tab[0], th)
        assert np.all(tab == tab[0])
    c = cai.cai_config_default(0, 1, 64, 256, 4096, 32, 4)   # t = 0: theta = theta_s = 0.9
    tab = cai.cai_test_theta_table(c, 0, 0)
    for p, r in _golden("position_factors.txt"):
        want = min(max(0.9 * float(r), 0.20), 0.98)
        assert abs(float(tab[int(p)]) - want) <= 1e-7, (p, tab[int(p)], want)


@pytest.mark.parametrize("flags", [0, 2, 2 | 8, 2 | 16, 2 | 32, 2 | 64, 1 | 2])
def test_theta_table_matches_oracle(flags):
    # Every position, block and step of several shapes against the oracle's
    # fp64 theta_i(t) rounded to fp32 (one rounding on each side).
    import oracle
    from tests import parity
    for P, T, nb in ((16, 8, 3), (32, 32, 8), (50, 20, 6), (64, 64, 16)):
        c = cai.cai_config_default(0, 2, P, 256, 4096, T, nb)
        c.flags = flags
        ocfg = parity.oracle_config(c)
        for blk in range(nb):
            for t in range(T):
                tab = cai.cai_test_theta_table(c, blk, t)
                want = np.array([oracle.theta_token(ocfg, blk + 1, t, p) for p in range(P)],
                                np.float32)
                ulp = np.spacing(want)
                assert np.all(np.abs(tab - want) <= ulp), (P, T, blk, t, flags)


def test_theta_table_arguments():
    c = cai.cai_config_default(0, 1, 16, 256, 4096, 8, 2)
    lib = cai.lib()
    out = np.zeros(16, np.float32)
    ptr = out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
    assert lib.cai_test_theta_table(ctypes.byref(c), 2, 0, ptr) == cai.CAI_ERR_ARG
    assert lib.cai_test_theta_table(ctypes.byref(c), 0, 8, ptr) == cai.CAI_ERR_ARG
    assert lib.cai_test_theta_table(ctypes.byref(c), -1, 0, ptr) == cai.CAI_ERR_ARG
    assert lib.cai_test_theta_table(None, 0, 0, ptr) == cai.CAI_ERR_ARG
    assert lib.cai_test_theta_table(ctypes.byref(c), 0, 0, None) == cai.CAI_ERR_ARG
    c.P = 0
    assert lib.cai_test_theta_table(ctypes.byref(c), 0, 0, ptr) == cai.CAI_ERR_SHAPE


def test_kernel_code_sha_follows_included_headers(tmp_path):
    # The bench reports a DRAM traffic record only while the kernel's code
    # still has the recorded sha: a code change in a header the kernel
    # includes (even indirectly) changes it, a comment edit does not.
    import bench
    (tmp_path / "a.cuh").write_text('#include "b.cuh"\nint a() { return b(); }\n')
    (tmp_path / "b.cuh").write_text('#include "c.cuh"\nint b() { return c(); }\n')
    (tmp_path / "c.cuh").write_text('#include "a.cuh"\nint c() { return 1; }  // one\n')
    s0 = bench.source_code_sha(str(tmp_path / "a.cuh"))
    (tmp_path / "c.cuh").write_text('#include "a.cuh"\n/* note */\nint c() { return 1; }  // two\n')
    assert bench.source_code_sha(str(tmp_path / "a.cuh")) == s0
    (tmp_path / "c.cuh").write_text('#include "a.cuh"\nint c() { return 2; }\n')
    assert bench.source_code_sha(str(tmp_path / "a.cuh")) != s0
