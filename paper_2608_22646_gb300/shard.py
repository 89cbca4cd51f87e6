"""Vocabulary-parallel decoding head across ranks (one shard context per rank).

Each rank holds the rows [v0, v0 + V_shard) of the LM-head weight in a shard
context (``cai_init_vocab_shard``) and a full copy of the controller state.
One denoising step is the shard's LM head (``cai_shard_head``: one 16-byte
triple per masked row, the argmax as a global vocabulary index), an
all-gather of every rank's triples over ``torch.distributed`` (NCCL between
GPUs; gloo works for CPU tensors), and the merge + commit on every rank
(``cai_shard_commit``), which leaves every rank with the same state.  Box 1's
maximum, sum of exponentials and lowest-index argmax are exact merges over
any split of the vocabulary, so the result is the unsharded head's.

Argument marshalling and the collective only: the head, the merge and the
commit run in the library's kernels.
"""
from __future__ import annotations

import paper_2608_22646_gb300 as cai


def vocab_slices(V: int, n_shards: int, granule: int = 256) -> list[tuple[int, int]]:
    """A split of V vocabulary rows into n_shards contiguous slices (v0, rows)
    whose sizes differ by at most one granule (the LM head's 256-row tile)."""
    if n_shards < 1 or V < n_shards:
        raise ValueError(f"cannot split {V} rows in {n_shards} shards")
    units = -(-V // granule)
    out = []
    for k in range(n_shards):
        a = min(V, (units * k // n_shards) * granule)
        b = min(V, (units * (k + 1) // n_shards) * granule)
        out.append((a, b - a))
    if any(n <= 0 for _, n in out):
        raise ValueError(f"{V} rows leave an empty shard among {n_shards}")
    return out


def exchange_triples(local, group=None):
    """All-gather of every rank's exchange buffer ([rows, 4] float32) into
    [world, rows, 4], rank k's buffer at index k."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    parts = [torch.empty_like(local) for _ in range(world)]
    dist.all_gather(parts, local.contiguous(), group=group)
    return torch.stack(parts)


class ShardStepper:
    """One rank's side of the vocabulary-parallel step: owns the rank's
    exchange buffer and runs head -> all-gather -> commit."""

    def __init__(self, ctx: cai.Ctx, group=None):
        import torch
        self.ctx = ctx
        self.group = group
        self.rows = cai.cai_shard_rows(ctx)
        self.local = torch.empty((self.rows, 4), dtype=torch.float32, device="cuda")

    def step(self, hidden, stream=None) -> None:
        cai.cai_shard_head(self.ctx, hidden, self.local, stream)
        gathered = exchange_triples(self.local, self.group)
        cai.cai_shard_commit(self.ctx, gathered, stream)
