"""Multi-GPU DP-SGD steps (one process per GPU), in the two partitions of the
step that need only one exchange each.

By example (``data_parallel_step``).  The batch is sharded by example: a
rank holds whole examples, every layer of them, so its per-example norms,
clip factors and clipped sums are local (Algorithm 2's per-example work needs
no other rank).  The exchange is the sum of the committed clipped sums,
done as a reduce-scatter of the flat parameter vector: each rank then holds
the summed commitment of one contiguous slice of the parameters, adds the
released noise of that slice only (the Philox stream is keyed by the global
parameter index, so a slice's noise is the same whichever rank makes it),
and an all-gather gives every rank the whole released gradient
out_scale (S + sigma C z).  Each rank's context is created for its own shard:
B = its example count (``shard_examples``) and out_scale = 1 / B_global for
the paper's average (or 1 for the sum), the same (C, sigma, seed, step)
everywhere.  Audit indices passed to ``dp_audit_emit`` are local; the global
index of local example i is ``start + i``.

By layer (``layer_parallel_step``).  Every rank holds all B examples but
only a contiguous range of the layers (``shard_layers``), its context
created with those layers and ``param_base`` = the parameters of the layers
before them.  ||g_i|| runs over every trainable parameter (Sec. 2.2), so the
only exchange is a sum all-reduce of the B partial squared norms before the
clip factors; the clipped sums and the noise of a rank's layers are then
local, and the noise keys are global indices by construction.

The library's calls are queued on the stream the collectives run on (create
the context with torch's current stream), so each collective orders after
the kernels that feed it and the next kernels after it.  ``host_staging``
runs the collectives on host copies (a gloo group with device tensors).
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


def shard_layers(shapes: Sequence[Sequence[int]], world: int, rank: int) -> Tuple[int, int, int]:
    """(first layer, layer count, param_base) of rank ``rank``'s contiguous
    range of layers: ranges balanced by parameter count (each rank at least
    one layer), param_base = the parameters of the layers before it."""
    L = len(shapes)
    if world < 1 or not 0 <= rank < world or L < world:
        raise ValueError(f"cannot shard {L} layers over {world} ranks (rank {rank})")
    sizes = [int(s[0]) * int(s[1]) for s in shapes]
    cum = [0]
    for n in sizes:
        cum.append(cum[-1] + n)
    # cut r: the layer boundary closest to r/world of the parameters, kept
    # so that every range holds at least one layer
    cuts = [0]
    for r in range(1, world):
        target = cum[-1] * r / world
        l = min(range(L + 1), key=lambda i: (abs(cum[i] - target), i))
        l = min(max(l, cuts[-1] + 1), L - (world - r))
        cuts.append(l)
    cuts.append(L)
    first, last = cuts[rank], cuts[rank + 1]
    return first, last - first, sum(sizes[:first])


class FlatOutputs:
    """Every layer's output [d_in][d_out] as a view of one fp32 vector in
    parameter order, so the global parameter index p of the noise is the
    offset in it.  The vector is padded with zeros to ``world`` equal slices
    of a multiple of 4 floats (each slice starts on a Philox quad and a
    16-byte boundary).  Every layer's size must be a multiple of 4 floats
    (16-byte aligned views)."""

    def __init__(self, shapes: Sequence[Sequence[int]], world: int, device=None):
        import torch
        sizes = [int(s[0]) * int(s[1]) for s in shapes]
        if any(n % 4 for n in sizes):
            raise ValueError("every layer's d_in * d_out must be a multiple of 4")
        self.P = sum(sizes)
        self.world = world
        self.chunk = -(-self.P // (4 * world)) * 4
        self.flat = torch.zeros(world * self.chunk, dtype=torch.float32, device=device)
        self._slice = None
        self.views = []
        off = 0
        for (i, o), n in zip(shapes, sizes):
            self.views.append(self.flat[off:off + n].view(int(i), int(o)))
            off += n

    def slice_buffer(self):
        """This rank's slice of the reduced vector (allocated once)."""
        import torch
        if self._slice is None:
            self._slice = torch.empty(self.chunk, dtype=self.flat.dtype, device=self.flat.device)
        return self._slice

    def slice_of(self, rank: int) -> Tuple[int, int]:
        """(first global index, parameter count) of rank's slice."""
        first = rank * self.chunk
        return first, max(0, min(self.chunk, self.P - first))


class _Comm:
    """The three collectives, on the tensors themselves or on host copies."""

    def __init__(self, group, host_staging: bool):
        import torch.distributed as dist
        self.dist, self.group, self.host = dist, group, host_staging

    def _run(self, fn, out, inp):
        if not self.host:
            fn(out, inp, group=self.group)
            return
        o, i = out.cpu(), inp.cpu()
        fn(o, i, group=self.group)
        out.copy_(o)

    def all_reduce(self, t):
        if not self.host:
            self.dist.all_reduce(t, op=self.dist.ReduceOp.SUM, group=self.group)
            return
        h = t.cpu()
        self.dist.all_reduce(h, op=self.dist.ReduceOp.SUM, group=self.group)
        t.copy_(h)

    def reduce_scatter(self, out, inp):
        self._run(lambda o, i, group: self.dist.reduce_scatter_tensor(
            o, i, op=self.dist.ReduceOp.SUM, group=group), out, inp)

    def all_gather(self, out, inp):
        self._run(self.dist.all_gather_into_tensor, out, inp)


def data_parallel_step(ctx: int, A_list, D_list, out: FlatOutputs, flags: int = 0, group=None,
                       lib=None, host_staging: bool = False) -> None:
    """One step of the batch sharded by example over ``group``: local norms,
    clip factors and noiseless clipped sums of every layer into
    ``out.views`` (the commitment), a reduce-scatter of ``out.flat``, the
    noise of this rank's slice, then an all-gather, after which every rank
    holds the released gradient in ``out.views``.  ``flags`` DP_NO_NOISE
    leaves the summed commitment.  ``lib`` defaults to this package's
    binding (tests pass a stand-in)."""
    import torch.distributed as dist

    if lib is None:
        import paper_2609_20532_gb300 as lib
    if flags & ~lib.DP_NO_NOISE:
        raise ValueError("data_parallel_step takes no flag but DP_NO_NOISE")
    comm = _Comm(group, host_staging)
    rank = dist.get_rank(group)
    if dist.get_world_size(group) != out.world:
        raise ValueError("FlatOutputs were laid out for another world size")
    layers = list(range(len(out.views)))
    lib.dp_layer_norms_batch(ctx, layers, A_list, D_list)
    lib.dp_clip_factors(ctx)
    lib.dp_clipped_sum_noise_batch(ctx, layers, A_list, D_list, out.views, lib.DP_NO_NOISE)
    mine = out.slice_buffer()
    comm.reduce_scatter(mine, out.flat)
    first, n = out.slice_of(rank)
    if not flags & lib.DP_NO_NOISE and n > 0:
        lib.dp_noise_add_range(ctx, first, n, mine)
    comm.all_gather(out.flat, mine)


def layer_parallel_step(ctx: int, A_list, D_list, outs, B: int, flags: int = 0, group=None,
                        lib=None, host_staging: bool = False, s_total=None) -> None:
    """One step of the model sharded by layer over ``group``: the norms of
    this rank's layers, the all-reduce of the B partial squared norms, the
    clip factors of the summed norms, then this rank's clipped sums and
    noise (``flags`` as dp_clipped_sum_noise: 0 or DP_NO_NOISE).  The
    context holds only this rank's layers, with their global param_base.
    ``s_total`` (optional, fp32 [B] on the device) receives the summed
    squared norms."""
    import torch

    if lib is None:
        import paper_2609_20532_gb300 as lib
    comm = _Comm(group, host_staging)
    layers = list(range(len(outs)))
    lib.dp_layer_norms_batch(ctx, layers, A_list, D_list)
    s = s_total if s_total is not None else torch.empty(B, dtype=torch.float32,
                                                         device=outs[0].device)
    lib.dp_partial_sqnorms(ctx, s)
    comm.all_reduce(s)
    lib.dp_clip_factors_from(ctx, s)
    lib.dp_clipped_sum_noise_batch(ctx, layers, A_list, D_list, outs, flags)
