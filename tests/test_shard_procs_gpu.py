"""The row-sharded dense step across processes: four gloo ranks on the one
GPU hold 1, 2, 4 or 8 shards between them (round-robin; a rank may hold
none), and exchange real blocks with torch.distributed: an all-reduce MAX of
the D + 1 exponent bytes, then an all-reduce SUM of the D + 1 fixed-point
words (Section 2.3: the statistics are sums of g^2, so the ranks need only
a kilobyte-scale exchange, and the result must be bitwise identical at any
world size).  Every rank also runs the whole-table ember_step_dense on the
same inputs and checks its shards' rows of W and r, and c, bit for bit;
rank 0 gates that whole-table step against the CPU oracle.

The kernels of different processes never wait on one another: the exchange
is on the host, between the launches.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

pytestmark = pytest.mark.gpu

WORLD = 4
V, D, STEPS = 3001, 1024, 3


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(WORLD), MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import sys
    here = os.path.dirname(os.path.abspath(__file__))
    sys.path.insert(0, here)
    sys.path.insert(0, os.path.dirname(here))
    import torch
    import torch.distributed as dist
    from paper_2607_01455_gb300.ember import Ember
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    result = {}
    try:
        for nshards in (1, 2, 4, 8):
            mine = [k for k in range(nshards) if k % WORLD == rank]
            ref = Ember(V, D, wdtype="bf16", device=dev)
            W0 = (torch.randn(V, D, generator=torch.Generator(device=dev).manual_seed(11), device=dev) * 0.02).to(
                torch.bfloat16)
            Wref = W0.clone()
            shards = {k: Ember(V, D, wdtype="bf16", device=dev) for k in mine}
            plan = {k: shards[k].shard_rows(k, nshards) for k in mine}
            Ws = {k: W0[r0:r0 + n].clone() for k, (r0, n) in plan.items()}
            exchanged = 0
            for t in range(1, STEPS + 1):
                g = torch.Generator(device=dev).manual_seed(500 + t)
                G = torch.randn(V, D, generator=g, device=dev) * 1e-3
                G *= torch.rand(V, 1, generator=g, device=dev) * 2 + 0.01
                if rank == 0 and nshards == 8 and t == STEPS:
                    from parity import Opt, gated_dense_step
                    gated_dense_step(ref, Wref, G, 1e-3, t, Opt())
                else:
                    ref.step_dense(Wref, G, 1e-3, t)
                Gs = {k: G[r0:r0 + n].contiguous() for k, (r0, n) in plan.items()}
                # first exchange: the largest exponent per column, all-reduced with MAX
                scales = torch.zeros(D + 1, dtype=torch.uint8, device=dev)
                for k in mine:
                    sk = torch.zeros(D + 1, dtype=torch.uint8, device=dev)
                    shards[k].shard_reduce(k, nshards, Gs[k], sk)
                    scales = torch.maximum(scales, sk)
                scales_h = scales.cpu()
                dist.all_reduce(scales_h, op=dist.ReduceOp.MAX)
                scales = scales_h.to(dev)
                # second exchange: the fixed-point totals, all-reduced with SUM
                sums = torch.zeros(D + 1, dtype=torch.int64, device=dev)
                for k in mine:
                    pk = torch.zeros(D + 1, dtype=torch.int64, device=dev)
                    shards[k].shard_pack(k, nshards, scales, pk)
                    sums += pk
                sums_h = sums.cpu()
                dist.all_reduce(sums_h, op=dist.ReduceOp.SUM)
                exchanged = scales_h.numel() * scales_h.element_size() + sums_h.numel() * sums_h.element_size()
                sums = sums_h.to(dev)
                for k in mine:
                    shards[k].shard_update(k, nshards, Ws[k], Gs[k], scales, sums, 1e-3, t)
            torch.cuda.synchronize()
            ok = True
            for k, (r0, n) in plan.items():
                ok &= torch.equal(Ws[k].view(torch.int16), Wref[r0:r0 + n].view(torch.int16))
                ok &= torch.equal(shards[k].r[r0:r0 + n].view(torch.int32), ref.r[r0:r0 + n].view(torch.int32))
                ok &= torch.equal(shards[k].c.view(torch.int32), ref.c.view(torch.int32))
                ok &= shards[k].device_status() == 0
            result[nshards] = (bool(ok), len(mine), exchanged)
            dist.barrier()
    except Exception as ex:  # reported to the parent, which fails the test
        result["error"] = repr(ex)
    finally:
        dist.destroy_process_group()
    out[rank] = result


def test_four_processes_exchange_kilobyte_blocks_bitwise(cuda_device):
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(_free_port(), out), nprocs=WORLD, join=True)
        res = dict(out)
    assert sorted(res) == list(range(WORLD))
    for rank, r in res.items():
        assert "error" not in r, (rank, r["error"])
        for nshards in (1, 2, 4, 8):
            ok, held, exchanged = r[nshards]
            assert ok, (rank, nshards)
            assert held == len([k for k in range(nshards) if k % WORLD == rank])
            assert exchanged == 9 * (D + 1)  # D + 1 bytes, then D + 1 words of 8 bytes
    assert np.all([res[k][8][1] == 2 for k in range(WORLD)])
