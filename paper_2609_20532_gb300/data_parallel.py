"""Data-parallel DP-SGD step over ranks (one process per GPU).

The batch is sharded by example: a rank holds whole examples, every layer of
them, so its per-example norms, clip factors and clipped sums are local
(Algorithm 2's per-example work needs no other rank).  The only exchange is
one sum all-reduce of the committed clipped sums.  The noise is added after
it, on every rank, from the same key: the Philox stream is keyed by the
global parameter index, so every rank generates the same z and all ranks end
the step holding the same released gradient out_scale (S + sigma C z).

Each rank's context is created for its own shard: B = its example count
(``shard_examples``) and out_scale = 1 / B_global for the paper's average
(or 1 for the sum), the same (C, sigma, seed, step) everywhere.  Audit
indices passed to ``dp_audit_emit`` are local; the global index of local
example i is ``start + i``.

The library's calls must be queued on the stream the collective runs on
(create the context with torch's current stream); the all-reduce then orders
after the clipped sums and the noise after the all-reduce.
"""

from __future__ import annotations

from typing import Optional, Sequence, Tuple


def shard_examples(B_global: int, world: int, rank: int) -> Tuple[int, int]:
    """(start, count) of the examples rank ``rank`` of ``world`` holds:
    contiguous blocks, the first B_global % world ranks one example more."""
    if world < 1 or not 0 <= rank < world or B_global < world:
        raise ValueError(f"cannot shard {B_global} examples over {world} ranks (rank {rank})")
    base, extra = divmod(B_global, world)
    start = rank * base + min(rank, extra)
    return start, base + (1 if rank < extra else 0)


def data_parallel_step(ctx: int, layers: Sequence[int], A_list, D_list, outs, flags: int = 0,
                       group=None, lib=None) -> None:
    """One step of the sharded batch: local norms, clip factors and noiseless
    clipped sums (the commitment), a sum all-reduce of ``outs`` over
    ``group``, then the released noise (unless ``flags`` holds DP_NO_NOISE,
    which leaves the reduced commitment).  ``outs`` are overwritten.
    ``lib`` defaults to this package's binding (tests pass a stand-in)."""
    import torch.distributed as dist

    if lib is None:
        import paper_2609_20532_gb300 as lib
    if flags & ~lib.DP_NO_NOISE:
        raise ValueError("data_parallel_step takes no flag but DP_NO_NOISE")
    layers = list(layers)
    lib.dp_layer_norms_batch(ctx, layers, A_list, D_list)
    lib.dp_clip_factors(ctx)
    lib.dp_clipped_sum_noise_batch(ctx, layers, A_list, D_list, outs, lib.DP_NO_NOISE)
    for o in outs:
        dist.all_reduce(o, op=dist.ReduceOp.SUM, group=group)
    if not flags & lib.DP_NO_NOISE:
        lib.dp_clipped_sum_noise_batch(ctx, layers, None, None, outs, lib.DP_NOISE_ONLY)
