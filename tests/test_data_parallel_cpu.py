"""Host logic of the data-parallel step on CPU (gloo, world size 2).

Each rank holds a contiguous shard of the batch.  In place of the CUDA
library each rank runs a stand-in whose calls compute what the library's
calls compute, with the oracle: local per-example norms and clip factors, the
noiseless clipped sum of its own examples (times out_scale), and the noise
added to the reduced sum.  After ``data_parallel_step`` every rank must hold
the single-process oracle step over the whole batch, with the noise added
once, and the DP_NO_NOISE variant the reduced commitment."""

import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SHAPES = [(6, 5), (5, 3)]
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

    def __init__(self, shapes, out_scale):
        from oracle import dp_oracle as O
        self.O = O
        self.out_scale = out_scale
        self.p_base = np.cumsum([0] + [i * o for i, o in shapes])[:-1]
        self.n = None
        self.c = None

    def dp_layer_norms_batch(self, ctx, layers, A_list, D_list):
        self.n = np.stack([self.O.layer_sqnorms(A, D) for A, D in zip(A_list, D_list)])

    def dp_clip_factors(self, ctx):
        _, self.c = self.O.clip_factors(self.n, C)

    def dp_clipped_sum_noise_batch(self, ctx, layers, A_list, D_list, outs, flags):
        for r, l in enumerate(layers):
            o = outs[r]
            if flags & self.DP_NOISE_ONLY:
                z = self.O.gaussian_noise(SEED, STEP, int(self.p_base[l]), o.numel())
                o += torch.from_numpy(self.out_scale * SIGMA * C * z.reshape(o.shape)).float()
            else:
                S = self.O.clipped_sum(A_list[r], D_list[r], self.c)
                o.copy_(torch.from_numpy(self.out_scale * S).float())


def _worker(rank, world, port, out, flags):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    from paper_2609_20532_gb300.data_parallel import data_parallel_step, shard_examples
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    start, count = shard_examples(B, world, rank)
    layers = _inputs()
    A = [a[start:start + count] for a, _ in layers]
    D = [d[start:start + count] for _, d in layers]
    outs = [torch.zeros(i, o) for i, o in SHAPES]
    lib = _OracleLib(SHAPES, out_scale=1.0 / B)
    data_parallel_step(None, range(len(SHAPES)), A, D, outs, flags=flags, lib=lib)
    out[rank] = ([o.numpy().copy() for o in outs], lib.c.copy(), start)
    dist.barrier()
    dist.destroy_process_group()


def _run(flags):
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out, flags)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    return [out[r] for r in range(world)]


@pytest.mark.parametrize("noise", [True, False])
def test_sharded_step_equals_whole_batch_step(noise):
    sys.path.insert(0, ROOT)
    from oracle import dp_oracle as O
    res = _run(0 if noise else 0x1)
    ref = O.dp_step(_inputs(), C, SIGMA, SEED, STEP, out_scale=1.0 / B, noise=noise)
    for outs, c, start in res:
        for o, r in zip(outs, ref["out"]):
            assert np.linalg.norm(o - r) <= 1e-6 * np.linalg.norm(r)
        # the clip factors are those of the rank's own examples
        assert np.allclose(c, ref["c"][start:start + len(c)], rtol=1e-12)
    # every rank ends the step with the same bits
    for a, b in zip(res[0][0], res[1][0]):
        assert np.array_equal(a, b)


def test_shard_examples():
    sys.path.insert(0, ROOT)
    from paper_2609_20532_gb300.data_parallel import shard_examples
    assert [shard_examples(7, 2, r) for r in range(2)] == [(0, 4), (4, 3)]
    assert [shard_examples(8, 4, r) for r in range(4)] == [(0, 2), (2, 2), (4, 2), (6, 2)]
    spans = [shard_examples(10, 3, r) for r in range(3)]
    assert spans == [(0, 4), (4, 3), (7, 3)]
    with pytest.raises(ValueError):
        shard_examples(1, 2, 0)
