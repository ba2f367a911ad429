"""Host logic of the two multi-GPU partitions on CPU (gloo, world size 2).

In place of the CUDA library each rank runs a stand-in whose calls compute
what the library's calls compute, with the oracle: per-example norms and
clip factors, noiseless clipped sums (times out_scale), the noise of a range
of global parameter indices, a context's partial squared norms and clip
factors from given totals.

By example: each rank holds a contiguous shard of the batch; after
``data_parallel_step`` (reduce-scatter of the flat commitment, noise of the
rank's own slice, all-gather) every rank must hold the single-process oracle
step over the whole batch, with every slice's noise added exactly once, and
the DP_NO_NOISE variant the summed commitment.

By layer: each rank holds all examples and a contiguous range of the layers;
after ``layer_parallel_step`` (all-reduce of the partial squared norms) the
clip factors are those of the whole model and each rank's outputs are the
whole-model oracle step's outputs for its layers (noise keyed by global
index through param_base)."""

import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SHAPES = [(6, 6), (5, 4), (4, 3), (2, 10)]
B, T = 7, 3
C, SIGMA, SEED, STEP = 0.4, 1.3, 11, 4


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _inputs():
    rng = np.random.default_rng(5)
    return [(rng.standard_normal((B, T, i)), 0.3 * rng.standard_normal((B, T, o)))
            for i, o in SHAPES]


class _OracleLib:
    """What one rank's library calls compute, written with the oracle."""

    DP_NO_NOISE, DP_NOISE_ONLY = 0x1, 0x2

    def __init__(self, shapes, out_scale, param_base=0):
        from oracle import dp_oracle as O
        self.O = O
        self.out_scale = out_scale
        self.p_base = param_base + np.cumsum([0] + [i * o for i, o in shapes])[:-1]
        self.n = None
        self.c = None

    def _noise(self, first, n):
        return self.out_scale * SIGMA * C * self.O.gaussian_noise(SEED, STEP, int(first), int(n))

    def dp_layer_norms_batch(self, ctx, layers, A_list, D_list):
        self.n = np.stack([self.O.layer_sqnorms(A, D) for A, D in zip(A_list, D_list)])

    def dp_clip_factors(self, ctx):
        _, self.c = self.O.clip_factors(self.n, C)

    def dp_partial_sqnorms(self, ctx, s):
        s.copy_(torch.from_numpy(self.n.sum(axis=0)).float())

    def dp_clip_factors_from(self, ctx, s):
        _, self.c = self.O.clip_factors(s.double().numpy()[None, :], C)

    def dp_noise_add_range(self, ctx, first, n, out):
        out[:n] += torch.from_numpy(self._noise(first, n)).float()

    def dp_clipped_sum_noise_batch(self, ctx, layers, A_list, D_list, outs, flags):
        for r, l in enumerate(layers):
            o = outs[r]
            if flags & self.DP_NOISE_ONLY:
                o += torch.from_numpy(self._noise(self.p_base[l], o.numel()).reshape(o.shape)).float()
                continue
            S = self.out_scale * self.O.clipped_sum(A_list[r], D_list[r], self.c)
            if not flags & self.DP_NO_NOISE:
                S = S + self._noise(self.p_base[l], o.numel()).reshape(o.shape)
            o.copy_(torch.from_numpy(S).float())


def _init(rank, world, port):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    return dist


def _worker_examples(rank, world, port, out, flags):
    dist = _init(rank, world, port)
    from paper_2609_20532_gb300.data_parallel import (FlatOutputs, data_parallel_step,
                                                      shard_examples)
    start, count = shard_examples(B, world, rank)
    layers = _inputs()
    A = [a[start:start + count] for a, _ in layers]
    D = [d[start:start + count] for _, d in layers]
    fo = FlatOutputs(SHAPES, world)
    lib = _OracleLib(SHAPES, out_scale=1.0 / B)
    noised = []
    real = lib.dp_noise_add_range
    lib.dp_noise_add_range = lambda ctx, first, n, o: (noised.append((first, n)),
                                                       real(ctx, first, n, o))
    data_parallel_step(None, A, D, fo, flags=flags, lib=lib)
    out[rank] = ([v.numpy().copy() for v in fo.views], lib.c.copy(), start, noised,
                 fo.flat[fo.P:].numpy().copy())
    dist.barrier()
    dist.destroy_process_group()


def _worker_layers(rank, world, port, out, flags):
    dist = _init(rank, world, port)
    from paper_2609_20532_gb300.data_parallel import layer_parallel_step, shard_layers
    first, count, pbase = shard_layers(SHAPES, world, rank)
    mine = SHAPES[first:first + count]
    layers = _inputs()[first:first + count]
    outs = [torch.zeros(i, o) for i, o in mine]
    lib = _OracleLib(mine, out_scale=1.0 / B, param_base=pbase)
    s = torch.zeros(B)
    layer_parallel_step(None, [a for a, _ in layers], [d for _, d in layers], outs, B,
                        flags=flags, lib=lib, s_total=s)
    out[rank] = ([o.numpy().copy() for o in outs], lib.c.copy(), first, s.numpy().copy())
    dist.barrier()
    dist.destroy_process_group()


def _run(worker, flags):
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    procs = [ctx.Process(target=worker, args=(r, world, port, out, flags)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    return [out[r] for r in range(world)]


@pytest.mark.parametrize("noise", [True, False])
def test_sharded_by_example_equals_whole_batch_step(noise):
    sys.path.insert(0, ROOT)
    from oracle import dp_oracle as O
    from paper_2609_20532_gb300.data_parallel import FlatOutputs
    res = _run(_worker_examples, 0 if noise else 0x1)
    ref = O.dp_step(_inputs(), C, SIGMA, SEED, STEP, out_scale=1.0 / B, noise=noise)
    for outs, c, start, noised, pad in res:
        for o, r in zip(outs, ref["out"]):
            assert np.linalg.norm(o - r) <= 1e-6 * np.linalg.norm(r)
        # the clip factors are those of the rank's own examples
        assert np.allclose(c, ref["c"][start:start + len(c)], rtol=1e-12)
        assert not pad.any()   # the padding past P stays zero
    # every rank ends the step with the same bits
    for a, b in zip(res[0][0], res[1][0]):
        assert np.array_equal(a, b)
    # each rank generated the noise of its own slice only, and the slices
    # cover [0, P) once
    fo = FlatOutputs(SHAPES, 2)
    if noise:
        assert [r[3] for r in res] == [[fo.slice_of(0)], [fo.slice_of(1)]]
        (f0, n0), (f1, n1) = fo.slice_of(0), fo.slice_of(1)
        assert f0 == 0 and f0 + n0 == f1 and f1 + n1 == fo.P
    else:
        assert all(r[3] == [] for r in res)


@pytest.mark.parametrize("noise", [True, False])
def test_sharded_by_layer_equals_whole_model_step(noise):
    sys.path.insert(0, ROOT)
    from oracle import dp_oracle as O
    res = _run(_worker_layers, 0 if noise else 0x1)
    ref = O.dp_step(_inputs(), C, SIGMA, SEED, STEP, out_scale=1.0 / B, noise=noise)
    seen = []
    for outs, c, first, s in res:
        # clip factors and squared norms of the whole model on every rank
        assert np.allclose(c, ref["c"], rtol=1e-6)
        assert np.allclose(s, ref["n"].sum(axis=0), rtol=1e-6)
        for k, o in enumerate(outs):
            r = ref["out"][first + k]
            assert np.linalg.norm(o - r) <= 1e-6 * np.linalg.norm(r)
            seen.append(first + k)
    assert sorted(seen) == list(range(len(SHAPES)))


def test_shard_examples():
    sys.path.insert(0, ROOT)
    from paper_2609_20532_gb300.data_parallel import shard_examples
    assert [shard_examples(7, 2, r) for r in range(2)] == [(0, 4), (4, 3)]
    assert [shard_examples(8, 4, r) for r in range(4)] == [(0, 2), (2, 2), (4, 2), (6, 2)]
    spans = [shard_examples(10, 3, r) for r in range(3)]
    assert spans == [(0, 4), (4, 3), (7, 3)]
    with pytest.raises(ValueError):
        shard_examples(1, 2, 0)


def test_shard_layers_and_flat_layout():
    sys.path.insert(0, ROOT)
    from paper_2609_20532_gb300.data_parallel import FlatOutputs, shard_layers
    llm = [(4096, 11008), (11008, 4096), (4096, 12288)]
    assert [shard_layers(llm, 2, r) for r in range(2)] == [(0, 2, 0), (2, 1, 2 * 4096 * 11008)]
    for world in (1, 2, 3, 4):
        spans = [shard_layers(SHAPES, world, r) for r in range(world)]
        # contiguous, every layer once, at least one layer each, param_base consistent
        assert spans[0][0] == 0 and all(n >= 1 for _, n, _ in spans)
        for (f0, n0, _), (f1, _, pb1) in zip(spans, spans[1:]):
            assert f0 + n0 == f1
            assert pb1 == sum(i * o for i, o in SHAPES[:f1])
        assert spans[-1][0] + spans[-1][1] == len(SHAPES)
    with pytest.raises(ValueError):
        shard_layers(SHAPES, 5, 0)
    fo = FlatOutputs(SHAPES, 3)
    assert fo.chunk % 4 == 0 and 3 * fo.chunk >= fo.P > 2 * fo.chunk - 4 * 3
    assert [v.shape for v in fo.views] == [torch.Size(s) for s in SHAPES]
    assert all(v.data_ptr() % 16 == 0 for v in fo.views)
    with pytest.raises(ValueError):
        FlatOutputs([(3, 3)], 2)
