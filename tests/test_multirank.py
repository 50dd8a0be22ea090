"""Multi-rank sharding on the CPU (gloo, world_size 2).

The op shards without a data-path collective: noise is a function of the
tensor-global element index, so a rank that owns a row range passes its
row_offset and produces exactly the rows of the unsharded result.  Here two gloo
ranks each run the oracle on their shard; rank 0 gathers and compares bit for
bit, and the max-over-ranks reduction used for timing is checked too.
"""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import workloads as WL
    from oracle import roi_oracle as O
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    rows, cols, N, M, tau = 12, 64, 2, 4, 0.7
    W, phi, dWm = WL.make_inputs(rows, cols, "normal", 31)
    per = rows // world
    r0 = rank * per
    sl = slice(r0, r0 + per)
    f = O.mask_fwd(phi.numpy()[sl], WL.bf16_bits(W)[sl], N, M, tau, 5, 2, tensor_id=1, row_offset=r0)
    b = O.mask_bwd(phi.numpy()[sl], WL.bf16_bits(W)[sl], WL.bf16_bits(dWm)[sl], N, M, tau, 5, 2,
                   tensor_id=1, row_offset=r0)
    mine = torch.from_numpy(np.concatenate([f["soft"].ravel(), b["dlogits"].ravel(),
                                            f["Wm"].astype(np.float64).ravel()]))
    gathered = [torch.zeros_like(mine) for _ in range(world)] if rank == 0 else None
    dist.gather(mine, gathered, dst=0)
    t = torch.tensor([float(rank + 1)])
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    if rank == 0:
        full_f = O.mask_fwd(phi.numpy(), WL.bf16_bits(W), N, M, tau, 5, 2, tensor_id=1)
        full_b = O.mask_bwd(phi.numpy(), WL.bf16_bits(W), WL.bf16_bits(dWm), N, M, tau, 5, 2, tensor_id=1)
        n = per * cols
        ok = True
        for k, g in enumerate(gathered):
            g = g.numpy()
            rs = slice(k * per, (k + 1) * per)
            ok &= np.array_equal(g[:n], full_f["soft"][rs].ravel())
            ok &= np.array_equal(g[n:2 * n], full_b["dlogits"][rs].ravel())
            ok &= np.array_equal(g[2 * n:], full_f["Wm"][rs].astype(np.float64).ravel())
        out.put((bool(ok), float(t.item())))
    dist.destroy_process_group()


def test_row_shards_on_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    ok, tmax = q.get(timeout=300)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert ok
    assert tmax == 2.0
