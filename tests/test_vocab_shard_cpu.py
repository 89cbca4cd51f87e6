"""The vocabulary-parallel head's exchange on two gloo ranks (CPU, no GPU).

Each rank holds one slice of the vocabulary.  Every step it computes its
slice's triple (max logit, sum of exponentials, lowest global argmax) for
every masked row with the oracle, the ranks exchange them through
``paper_2608_22646_gb300.shard.exchange_triples`` (the all-gather the GPU path
uses), and every rank merges all slices and runs the controller.  Both ranks
must end with the same state, equal to the single-process trajectory over the
whole vocabulary; the exchange must keep rank order.  The CUDA merge and
commit of the same exchange are checked on the GPU (test_vocab_shard_gpu.py).
"""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2608_22646_gb300.shard import vocab_slices

V, H, B, P, T, NB = 4096, 256, 3, 16, 8, 2


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _inputs():
    import synth
    wl = synth.Workload("shards", B=B, H=H, V=V, gen_len=P * NB, P=P, T=T, a0="u04")
    W = synth.lm_head_weight(V, H, seed=77)
    return W, synth.HiddenStates(wl, W, "calibrated", seed=5)


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from paper_2608_22646_gb300.shard import exchange_triples
    W, hs = _inputs()
    Wb = oracle.bf16_bits(W)
    v0, n = vocab_slices(V, world)[rank]
    cfg = oracle.Config(B=B, P=P, T=T, n_blocks=NB)
    st = oracle.State(cfg)
    rows_cap = -(-B * P // 16) * 16
    order_ok = True
    for blk in range(NB):
        for t in range(T):
            hb = oracle.bf16_bits(hs(blk, t)).reshape(B, P, H)
            mk = st.masked(blk)
            rows = np.ascontiguousarray(hb[mk])
            M = rows.shape[0]
            local = torch.zeros((rows_cap, 4), dtype=torch.float64)
            local[:, 0] = -np.inf
            local[:, 2] = np.iinfo(np.int32).max
            if M:
                part = oracle.head_rows_shard(Wb[v0:v0 + n], rows, v0, n_threads=2)
                local[:M, 0] = torch.from_numpy(part["m"])
                local[:M, 1] = torch.from_numpy(part["S"])
                local[:M, 2] = torch.from_numpy(part["idx"].astype(np.float64))
            gathered = exchange_triples(local)
            order_ok &= bool(torch.equal(gathered[rank], local))
            conf = np.zeros((B, P))
            idx = np.full((B, P), -1, np.int32)
            if M:
                g = gathered[:, :M].numpy()
                merged = oracle.merge_shards([{"m": g[k, :, 0], "S": g[k, :, 1],
                                               "idx": g[k, :, 2].astype(np.int64)}
                                              for k in range(world)])
                conf[mk], idx[mk] = merged["conf"], merged["idx"]
            oracle.controller_step(st, blk, t, conf, idx)
            if np.all(st.exit_reason[:, blk] != 0):
                break
    q.put((rank, order_ok, {f: getattr(st, f) for f in oracle.State.FIELDS}))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_vocab_shards_match_the_full_vocabulary():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted((q.get(timeout=300) for _ in range(world)), key=lambda x: x[0])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert all(ok for _, ok, _ in out)
    import oracle
    W, hs = _inputs()
    full = oracle.run_trajectory(oracle.Config(B=B, P=P, T=T, n_blocks=NB), W, hs)
    for _, _, st in out:
        for f in ("tok", "cstep", "budget", "cand", "ell", "eta", "exit_reason", "exit_step",
                  "unresolved"):
            assert np.array_equal(st[f], getattr(full, f)), f
        np.testing.assert_allclose(st["conf"], full.conf, rtol=1e-12, atol=1e-15)
    assert (full.tok != -1).sum() > B * P      # the trajectory commits tokens in both blocks


def test_vocab_slices_cover_the_vocabulary():
    for V_, g in ((126464, 2), (126464, 4), (152064, 8), (1000, 3), (256, 1), (4097, 4)):
        sl = vocab_slices(V_, g)
        assert sl[0][0] == 0 and sum(n for _, n in sl) == V_
        assert all(a + n == b for (a, n), (b, _) in zip(sl[:-1], sl[1:]))
        assert max(n for _, n in sl) - min(n for _, n in sl) <= 256
