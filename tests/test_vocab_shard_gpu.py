"""The vocabulary-parallel head on one GPU: g shard contexts (each holding one
slice of W) run every step as shard head -> exchange -> merge + commit, the
exchange being the stack of the g exchange buffers (what the all-gather
produces across g GPUs).  Every step is checked teacher-forced against the
fp64 oracle over the whole vocabulary, and every shard's state must equal
every other's bit for bit."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests import parity

import paper_2608_22646_gb300 as cai
from paper_2608_22646_gb300.shard import vocab_slices

pytestmark = pytest.mark.gpu

FIELDS = ("tok", "conf", "s0", "budget", "cstep", "cand", "ell", "eta", "exit_reason",
          "exit_step", "unresolved", "m_hist")


def _shard_ctxs(cfg, W, g):
    ctxs = []
    for v0, n in vocab_slices(W.shape[0], g):
        ctxs.append(cai.cai_init_vocab_shard(cfg, W[v0:v0 + n].contiguous(), v0))
    return ctxs


def _step(ctxs, bufs, h):
    for c, b in zip(ctxs, bufs):
        cai.cai_shard_head(c, h, b)
    gathered = torch.stack(bufs)
    for c in ctxs:
        cai.cai_shard_commit(c, gathered)


@pytest.mark.parametrize("g,shape", [
    # (B, P, H, V, T, n_blocks): B P = 16 (a single-kernel shape unsharded),
    # B P = 320 (one and two row tiles, swapped and unswapped pair steps), a
    # vocabulary whose shards are not multiples of 256, and the batched layout.
    (2, (1, 16, 256, 4096, 8, 2)),
    (4, (1, 16, 256, 4096, 8, 2)),
    (2, (5, 64, 256, 4096, 10, 2)),
    (4, (5, 64, 256, 4096, 10, 2)),
    (3, (3, 32, 128, 5000, 8, 2)),
    (4, (64, 32, 256, 4096, 12, 2)),
])
def test_vocab_shards_match_full_vocabulary(g, shape):
    B, P, H, V, T, nb = shape
    wl = synth.Workload("shards", B=B, H=H, V=V, gen_len=P * nb, P=P, T=T, a0="u04")
    W = synth.lm_head_weight(V, H, device="cuda")
    hs = synth.HiddenStates(wl, W, "calibrated", seed=B * 7 + g)
    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, B, P, H, V, T, nb)
    ctxs = _shard_ctxs(cfg, W, g)
    ocfg = parity.oracle_config(cfg)
    W_host = oracle.bf16_bits(W)
    rep = parity.StepReport()
    try:
        rows = cai.cai_shard_rows(ctxs[0])
        assert rows == -(-B * P // 16) * 16
        bufs = [torch.empty((rows, 4), dtype=torch.float32, device="cuda") for _ in ctxs]
        pre = cai.cai_state_download(ctxs[0])
        for blk in range(nb):
            if blk:
                for c in ctxs:
                    cai.cai_block_advance(c)
            for t in range(T):
                h = hs(blk, t)
                _step(ctxs, bufs, h)
                torch.cuda.synchronize()
                posts = [cai.cai_state_download(c) for c in ctxs]
                for p in posts[1:]:
                    for f in FIELDS:
                        assert np.array_equal(p[f], posts[0][f]), (f, blk, t)
                parity.check_step(ocfg, W_host, h, pre, posts[0], blk, t, rep)
                pre = posts[0]
                if np.all(pre["exit_reason"][:, blk] != 0):
                    assert all(cai.cai_poll(c, 0, 5000) for c in ctxs)
                    break
        assert rep.rows >= B * P * nb
        assert all(cai.cai_test_check_guards(c) == 0 for c in ctxs)
    finally:
        for c in ctxs:
            cai.cai_free(c)


def test_vocab_shards_tie_across_the_boundary_takes_the_lower_index():
    # Rows 100 and 3000 of W are equal; they sit in different shards (slices
    # [0, 2048) and [2048, 4096)).  Hidden rows along W[100] make both logits
    # the maximum: the merged argmax is 100, the lower index, and c ~ 1/2.
    B, P, H, V, T = 1, 16, 256, 4096, 4
    W = synth.lm_head_weight(V, H, device="cuda")
    W[3000] = W[100]
    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, B, P, H, V, T, 1)
    ctxs = _shard_ctxs(cfg, W, 2)
    assert vocab_slices(V, 2)[1][0] == 2048
    try:
        rows = cai.cai_shard_rows(ctxs[0])
        bufs = [torch.empty((rows, 4), dtype=torch.float32, device="cuda") for _ in ctxs]
        scale = torch.linspace(300.0, 500.0, P, device="cuda")[:, None]
        h = (W[100].float()[None, :] * scale).to(torch.bfloat16).reshape(B, P, H)
        _step(ctxs, bufs, h)
        torch.cuda.synchronize()
        # each shard's own triple: shard 0 finds 100, shard 1 finds 3000 (global)
        assert np.all(bufs[0][:P, 2].view(torch.int32).cpu().numpy() == 100)
        assert np.all(bufs[1][:P, 2].view(torch.int32).cpu().numpy() == 3000)
        assert torch.equal(bufs[0][:P, 0], bufs[1][:P, 0])      # the same maximum, bit for bit
        o = oracle.head_rows(W, h.reshape(P, H))
        assert np.all(o["idx"] == 100)
        for c in ctxs:
            st = cai.cai_state_download(c)
            assert np.all(st["cand"][0, :P] == 100)
            np.testing.assert_allclose(st["s0"][0, :P], o["conf"], rtol=0, atol=parity.CONF_TOL)
        # rows past M carry the empty triple
        if rows > P:
            e = bufs[0][P:]
            assert torch.all(e[:, 1] == 0) and torch.all(e[:, 2].view(torch.int32) == 2**31 - 1)
    finally:
        for c in ctxs:
            cai.cai_free(c)


def test_vocab_shard_arguments_and_order():
    V, H, B, P, T = 4096, 256, 1, 16, 4
    W = synth.lm_head_weight(V, H, device="cuda")
    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, B, P, H, V, T, 2)
    big = torch.zeros((3000, H), dtype=torch.bfloat16, device="cuda")
    for Ws, v0 in ((W[:2048], -1), (big, 2000), (W[:32], 0)):   # v0 < 0, past V, < 64 rows
        with pytest.raises(cai.CaiError) as e:
            cai.cai_init_vocab_shard(cfg, Ws.contiguous(), v0)
        assert e.value.status == cai.CAI_ERR_SHAPE
    ctx = cai.cai_init_vocab_shard(cfg, W[:2048].contiguous(), 0)
    plain = cai.cai_init(cfg, W)
    try:
        h = torch.zeros((B, P, H), dtype=torch.bfloat16, device="cuda")
        buf = torch.empty((cai.cai_shard_rows(ctx), 4), dtype=torch.float32, device="cuda")
        with pytest.raises(cai.CaiError) as e:          # the plain step calls refuse a shard
            cai.cai_first_step(ctx, h)
        assert e.value.status == cai.CAI_ERR_ARG
        with pytest.raises(cai.CaiError) as e:          # and the shard calls a plain context
            cai.cai_shard_head(plain, h, buf)
        assert e.value.status == cai.CAI_ERR_ARG
        with pytest.raises(cai.CaiError) as e:          # commit before any head
            cai.cai_shard_commit(ctx, buf[None])
        assert e.value.status == cai.CAI_ERR_ORDER
        with pytest.raises(cai.CaiError) as e:          # host memory as the exchange buffer
            cai.cai_shard_head(ctx, h, buf.cpu())
        assert e.value.status == cai.CAI_ERR_ARG
        cai.cai_shard_head(ctx, h, buf)
        with pytest.raises(cai.CaiError) as e:          # a second head before the commit
            cai.cai_shard_head(ctx, h, buf)
        assert e.value.status == cai.CAI_ERR_ORDER
        with pytest.raises(cai.CaiError) as e:
            cai.cai_block_advance(ctx)
        assert e.value.status == cai.CAI_ERR_ORDER
        cai.cai_shard_commit(ctx, buf[None])
        torch.cuda.synchronize()
        st = cai.cai_get_stats(ctx)
        assert st["steps"] == 1 and st["kernels_per_step"] >= 5
    finally:
        cai.cai_free(ctx)
        cai.cai_free(plain)


@pytest.mark.parametrize("g", [2, 3])
def test_vocab_shards_full_size_llada(g):
    # The LLaDA-8B shape (V = 126464, H = 4096, B = 1, P = 32) split over g
    # shard contexts on one GPU, the first two blocks: every step checked at
    # the controller level (the oracle's Algorithm 1 on the merged triples the
    # shards produced, every integer field bit-exact), the shards' states
    # identical, and at step zero of each block 8 sampled rows recomputed by
    # the fp64 oracle over the whole vocabulary.
    wl = synth.WORKLOADS["llada"]
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device="cuda")
    hs = synth.HiddenStates(wl, W, "calibrated")
    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    ctxs = _shard_ctxs(cfg, W, g)
    ocfg = parity.oracle_config(cfg)
    W_host = oracle.bf16_bits(W)
    rng = np.random.default_rng(g)
    try:
        rows = cai.cai_shard_rows(ctxs[0])
        bufs = [torch.empty((rows, 4), dtype=torch.float32, device="cuda") for _ in ctxs]
        pre = cai.cai_state_download(ctxs[0])
        decoded = 0
        for blk in range(2):
            if blk:
                for c in ctxs:
                    cai.cai_block_advance(c)
            for t in range(wl.T):
                h = hs(blk, t)
                _step(ctxs, bufs, h)
                torch.cuda.synchronize()
                posts = [cai.cai_state_download(c) for c in ctxs]
                for p in posts[1:]:
                    for f in FIELDS:
                        assert np.array_equal(p[f], posts[0][f]), (f, blk, t)
                masked = np.argwhere(parity.to_oracle_state(ocfg, pre).masked(blk))
                decoded += parity.check_controller_step(ocfg, pre, posts[0], blk, t)
                if t == 0:
                    pick = rng.choice(len(masked), size=8, replace=False)
                    parity.check_rows_sampled(W_host, h, posts[0], blk,
                                              [tuple(masked[i]) for i in pick], wl.P)
                pre = posts[0]
                if np.all(pre["exit_reason"][:, blk] != 0):
                    break
        assert decoded >= 2 * wl.P
        assert np.all(pre["exit_reason"][:, :2] != 0)
    finally:
        for c in ctxs:
            cai.cai_free(c)
