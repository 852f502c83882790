"""Host side of the row-sharded dense step, on the CPU (no kernel runs).

The shard plan (which rows each shard holds, how big its exchange blocks
are) is host logic of the library: it must tile the table exactly at the
whole-table step's CTA row boundaries, give every shard blocks of the same
size (what an all-reduce needs: D + 1 exponent bytes and D + 1 fixed-point
words, kilobytes rather than the per-CTA partial rows), and reject bad
arguments before any CUDA call.  The last test runs the plan on world_size
3 gloo ranks and all-gathers it, as ranks of a sharded job would.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2607_01455_gb300 import ember as E
from paper_2607_01455_gb300.build import build_library


@pytest.fixture(scope="module", autouse=True)
def built():
    build_library()


def cta_rows(V, D):
    """Row boundaries of the whole-table step's CTAs: one per 4096 elements
    of G, at most 304 (two per SM of the GB300) and at most one per row."""
    nparts = max(1, min(V, 304, -(-V * D // 4096)))
    return [b * V // nparts for b in range(nparts + 1)]


@pytest.mark.parametrize("V,D", [(1, 16), (7, 16), (303, 16), (304, 2048), (305, 4096), (1000, 16),
                                 (1000, 200), (128256, 16), (128256, 8192)])
@pytest.mark.parametrize("n", [1, 2, 3, 4, 8, 300, 305])
def test_shards_tile_the_table_at_cta_boundaries(V, D, n):
    h = E.ember_create(V, D)
    try:
        bounds = set(cta_rows(V, D))
        nxt = 0
        for k in range(n):
            row0, rows = E.ember_shard_rows(h, k, n)
            assert row0 == nxt and rows >= 0
            assert row0 in bounds and row0 + rows in bounds
            nxt = row0 + rows
        assert nxt == V
        # the two blocks every shard all-reduces: one byte and one 64-bit word
        # per column, and one of each for the sums of r
        assert E.ember_shard_scale_bytes(h) == D + 1
        assert E.ember_shard_exchange_bytes(h) == 8 * (D + 1)
    finally:
        E.ember_destroy(h)


def test_exchange_is_kilobytes_at_the_lm_head_width():
    """Section 2.3 asks for a kilobyte-scale exchange: at D = 8192 the
    fixed-point block is 64 KiB and the exponent block 8 KiB."""
    h = E.ember_create(128256, 8192)
    try:
        assert E.ember_shard_exchange_bytes(h) == 65544
        assert E.ember_shard_scale_bytes(h) == 8193
    finally:
        E.ember_destroy(h)


def test_shard_rejects_on_host():
    lib = E.lib()
    h = E.ember_create(1000, 64)
    try:
        fake = 1 << 20
        import ctypes
        r0 = ctypes.c_int64(0)
        assert lib.ember_shard_rows(h, 2, 2, ctypes.byref(r0)) == -1
        assert lib.ember_shard_rows(h, -1, 2, ctypes.byref(r0)) == -1
        assert lib.ember_shard_rows(h, 0, 0, ctypes.byref(r0)) == -1
        assert lib.ember_shard_rows(None, 0, 1, ctypes.byref(r0)) == -1
        assert lib.ember_shard_exchange_bytes(None) == 0
        assert lib.ember_shard_scale_bytes(None) == 0
        red = lib.ember_shard_reduce
        assert red(h, 0, 2, fake, fake, fake, None) == E.EMBER_ERR_WORKSPACE
        assert red(h, 3, 2, fake, fake, fake, None) == E.EMBER_ERR_INVALID_ARG
        assert red(h, 0, 2, fake + 4, fake, fake, None) == E.EMBER_ERR_ALIGNMENT
        assert red(h, 0, 2, fake, fake + 2, fake, None) == E.EMBER_ERR_ALIGNMENT
        assert red(h, 0, 2, None, fake, fake, None) == E.EMBER_ERR_WORKSPACE  # checked after the plan
        assert red(h, 0, 2, fake, fake, None, None) == E.EMBER_ERR_INVALID_ARG
        pk = lib.ember_shard_pack
        assert pk(h, 0, 2, fake, fake, None) == E.EMBER_ERR_WORKSPACE
        assert pk(h, 0, 2, None, fake, None) == E.EMBER_ERR_INVALID_ARG
        assert pk(h, 0, 2, fake, None, None) == E.EMBER_ERR_INVALID_ARG
        assert pk(h, 0, 2, fake, fake + 4, None) == E.EMBER_ERR_ALIGNMENT
        assert pk(h, 2, 2, fake, fake, None) == E.EMBER_ERR_INVALID_ARG
        up = lib.ember_shard_update
        assert up(h, 0, 2, fake, fake, fake, fake, fake, 1e-3, 0, None) == E.EMBER_ERR_INVALID_ARG
        assert up(h, 0, 2, fake, fake, fake, fake, fake, float("nan"), 1, None) == E.EMBER_ERR_INVALID_ARG
        assert up(h, 0, 2, fake, fake, fake, None, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert up(h, 0, 2, fake, fake, fake, fake, fake + 4, 1e-3, 1, None) == E.EMBER_ERR_ALIGNMENT
        assert up(h, 0, 2, fake, fake, fake, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_WORKSPACE
    finally:
        E.ember_destroy(h)
    hp = E.ember_hparams_default()
    hp.variant = E.EMBER_VARIANT_ROW
    h = E.ember_create(1000, 64, hp)
    try:
        assert E.lib().ember_shard_reduce(h, 0, 2, 1 << 20, 1 << 20, 1 << 20, None) == E.EMBER_ERR_UNSUPPORTED
    finally:
        E.ember_destroy(h)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, V, D, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    h = E.ember_create(V, D)
    row0, rows = E.ember_shard_rows(h, rank, world)
    nbytes = E.ember_shard_exchange_bytes(h)
    E.ember_destroy(h)
    mine = torch.tensor([row0, rows, nbytes], dtype=torch.int64)
    parts = [torch.zeros(3, dtype=torch.int64) for _ in range(world)]
    dist.all_gather(parts, mine)
    dist.destroy_process_group()
    out[rank] = [p.tolist() for p in parts]


def test_three_gloo_ranks_agree_on_the_plan():
    world, port, V, D = 3, _free_port(), 1000, 200
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, V, D, out), nprocs=world, join=True)
        plans = dict(out)
    assert plans[0] == plans[1] == plans[2]
    rows = plans[0]
    assert rows[0][0] == 0 and sum(r[1] for r in rows) == V
    assert all(rows[k][0] + rows[k][1] == rows[k + 1][0] for k in range(world - 1))
    assert len({r[2] for r in rows}) == 1
