"""Sparse Ember step on the GPU (Section 2.2) against the CPU oracle.

The sparse step must equal the dense step of Algorithm 1 on the V x D
gradient whose row u is the sum of the per-occurrence rows of token u.  The
dedup (distinct ids and their counts) must match the oracle bit for bit;
untouched rows of W must stay bit-identical; W and the state must match the
oracle within the dense bar (1e-5 relative on the fp32 state, 1 bf16 ulp).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01455_gb300 import synth
from paper_2607_01455_gb300.ember import (EMBER_ERR_ID_OUT_OF_RANGE, EMBER_ERR_WORKSPACE, Ember,
                                          EmberError)
from parity import Opt, check_state, check_weights, oracle_kwargs, w_to_host

pytestmark = pytest.mark.gpu


def make(V, D, wdtype, max_N, opt=None):
    opt = opt or Opt()
    return Ember(V, D, wdtype=wdtype, beta2=opt.beta2, eps=opt.eps, maximize=opt.maximize,
                 bias_correction=opt.bias_correction, variant=opt.variant, max_sparse_N=max_N)


def batch(V, D, N, t, device, seed=0, zipf=1.1, std=1e-4):
    g = torch.Generator(device=device)
    g.manual_seed(seed * 1_000_003 + t)
    p = (torch.arange(V, device=device, dtype=torch.float64) + 1) ** -zipf
    cdf = torch.cumsum(p, 0)
    cdf /= cdf[-1].clone()
    u = torch.rand(N, generator=g, device=device, dtype=torch.float64)
    ids = torch.searchsorted(cdf, u, right=True).clamp_(max=V - 1).to(torch.int64)
    rows = torch.randn(N, D, generator=g, device=device) * std
    return ids, rows


def gated_sparse_step(emb, W, ids, rows, lr, t, opt):
    V = emb.V
    W0 = w_to_host(W)
    st0 = emb.state.cpu().numpy().copy()
    emb.step_sparse(W, ids, rows, lr, t)
    torch.cuda.synchronize()
    r, c = st0[:V].copy(), st0[V:].copy()
    Wo = W0.copy()
    oracle.step_sparse(Wo, ids.cpu().numpy().astype(np.int64), rows.cpu().numpy(), r, c,
                       float(np.float32(lr)), t, **oracle_kwargs(opt))
    st = emb.state.cpu().numpy()
    check_state(st[:V], r, "r")
    check_state(st[V:], c, "c")
    Wg = w_to_host(W)
    check_weights(Wg, Wo, lr, prev=W0, record=True, summed_input=True)
    # rows whose id does not occur keep their weights bit for bit
    touched = np.zeros(V, bool)
    ids_h = ids.cpu().numpy().astype(np.int64)
    touched[ids_h[(ids_h >= 0) & (ids_h < V)]] = True
    assert np.array_equal(Wg[~touched], W0[~touched])
    return touched


def check_dedup(emb, ids):
    uniq, counts = emb.unique(ids)
    want_u, want_c = oracle.dedup(ids.cpu().numpy().astype(np.int64), emb.V)
    np.testing.assert_array_equal(uniq.cpu().numpy(), want_u)
    np.testing.assert_array_equal(counts.cpu().numpy(), want_c)


# 1024-key sort tiles: 4096, 4097, 32768, 32769, 65536 and 65537 sit on tile
# edges; the largest batch spans 98 tiles.
@pytest.mark.parametrize("V,D,N", [
    (50, 8, 1), (50, 8, 37), (1000, 64, 4096), (1000, 64, 4097), (5000, 200, 9000),
    (3000, 203, 5000), (262144, 128, 12288), (100, 2048, 3000), (20000, 8192, 700),
    (262144, 8, 32768), (7, 8, 32768), (70000, 8, 32769), (5000, 8, 65536), (300000, 16, 50000),
    (5000, 8, 65537), (400000, 8, 100000),
])
@pytest.mark.parametrize("idtype", [torch.int64, torch.int32])
def test_dedup_bit_exact(cuda_device, V, D, N, idtype):
    emb = make(V, D, "bf16", N)
    ids, _ = batch(V, 1, N, 1, cuda_device, seed=V + N)
    check_dedup(emb, ids.to(idtype))
    # the map of touched rows is cleared afterwards: a step still matches
    W = torch.zeros(V, D, device=cuda_device, dtype=torch.bfloat16)
    ids2, rows2 = batch(V, D, N, 2, cuda_device, seed=V)
    gated_sparse_step(emb, W, ids2.to(idtype), rows2, 1e-3, 1, Opt())


@pytest.mark.parametrize("V,D,N", [
    (64, 4, 100), (1000, 64, 512), (1000, 203, 3000), (4096, 256, 8192),
    (30000, 896, 6000), (2000, 2048, 5000),
    # two column slices of the segment sums, the second 8 columns wide
    # (1032 = 1024 + 8), and bf16 rows that do not start on 16-byte
    # boundaries (1100 = 8 * 137 + 4)
    (1500, 1032, 2500), (3000, 1100, 4000),
])
@pytest.mark.parametrize("wdtype", ["bf16", "f32"])
def test_sparse_parity(cuda_device, V, D, N, wdtype):
    opt = Opt()
    emb = make(V, D, wdtype, N)
    g = torch.Generator(device=cuda_device)
    g.manual_seed(V)
    W = (torch.randn(V, D, generator=g, device=cuda_device) * 0.02).to(
        torch.bfloat16 if wdtype == "bf16" else torch.float32)
    for t in range(1, 4):
        ids, rows = batch(V, D, N, t, cuda_device, seed=D)
        gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)


@pytest.mark.parametrize("opt", [Opt(maximize=True), Opt(variant="row"), Opt(variant="col"),
                                 Opt(bias_correction=False), Opt(beta2=0.9, eps=1e-6)],
                         ids=["maximize", "row_only", "col_only", "no_bc", "beta2_0.9"])
def test_sparse_parity_hyperparameters(cuda_device, opt):
    V, D, N = 2000, 256, 3000
    emb = make(V, D, "bf16", N, opt)
    W = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    for t in range(1, 4):
        ids, rows = batch(V, D, N, t, cuda_device, seed=5)
        gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)


def test_sparse_equals_dense_on_scatter_summed_gradient(cuda_device):
    """Section 2.2: the sparse step is the dense step on the summed rows.
    Gated like the oracle comparisons: each step both paths start from the
    sparse path's W and state."""
    V, D, N = 3000, 512, 10000
    es, ed = make(V, D, "bf16", N), make(V, D, "bf16", 0)
    W0 = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    Ws, Wd = W0.clone(), W0.clone()
    for t in range(1, 4):
        ids, rows = batch(V, D, N, t, cuda_device, seed=9)
        G = torch.zeros(V, D, device=cuda_device, dtype=torch.float64)
        G.index_add_(0, ids, rows.double())
        Wd.copy_(Ws)
        ed.state.copy_(es.state)
        es.step_sparse(Ws, ids, rows, 1e-3, t)
        ed.step_dense(Wd, G.float(), 1e-3, t)
        torch.cuda.synchronize()
        check_state(es.state.cpu().numpy(), ed.state.cpu().numpy(), "state")
        check_weights(w_to_host(Ws), w_to_host(Wd), 1e-3, summed_input=True)


def test_sparse_edge_cases(cuda_device):
    V, D = 500, 64
    opt = Opt()
    emb = make(V, D, "bf16", 20000)
    W = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    t = 0
    # N = 0: every row of r decays, W does not move
    t += 1
    ids, rows = batch(V, D, 200, t, cuda_device)
    gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)
    t += 1
    W_before = W.clone()
    gated_sparse_step(emb, W, ids[:0], rows[:0], 1e-3, t, opt)
    assert torch.equal(W.view(torch.int16), W_before.view(torch.int16))
    # one id repeated across many tiles and chunks
    t += 1
    ids = torch.full((20000,), 7, dtype=torch.int64, device=cuda_device)
    rows = torch.randn(20000, D, device=cuda_device) * 1e-4
    gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)
    check_dedup(emb, ids)
    # every id distinct, in descending order
    t += 1
    ids = torch.arange(V - 1, -1, -1, device=cuda_device)
    rows = torch.randn(V, D, device=cuda_device) * 1e-4
    gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)
    # ids outside [0, V) are skipped and flagged; the rest is exact
    t += 1
    ids, rows = batch(V, D, 3000, t, cuda_device)
    ids[::97] = V
    ids[5] = -1
    ids[6] = 1 << 40
    gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)
    assert emb.device_status() == EMBER_ERR_ID_OUT_OF_RANGE
    assert emb.device_status() == 0  # reading the flag clears it
    # more ids than the workspace was bound for
    big = torch.zeros(20001, dtype=torch.int64, device=cuda_device)
    with pytest.raises(EmberError) as ex:
        emb.step_sparse(W, big, torch.zeros(20001, D, device=cuda_device), 1e-3, t + 1)
    assert ex.value.status == EMBER_ERR_WORKSPACE


def test_skipped_ids_leave_the_step_bit_identical(cuda_device):
    """The same batch, and the batch followed by 10000 skipped ids (id -1,
    whose rows are never read), give bit-identical W and state: skipped ids
    sort after every valid one, so the segment sums see the same order."""
    V, D, N, Npad = 20000, 256, 30000, 40000
    ids, rows = batch(V, D, N, 1, cuda_device, seed=11)
    ids_pad = torch.cat([ids, torch.full((Npad - N,), -1, dtype=ids.dtype, device=cuda_device)])
    rows_pad = torch.cat([rows, torch.full((Npad - N, D), float("nan"), device=cuda_device)])
    outs = []
    for i, r in ((ids, rows), (ids_pad, rows_pad)):
        emb = make(V, D, "bf16", Npad)
        W = (torch.randn(V, D, device=cuda_device, generator=torch.Generator(device=cuda_device)
                         .manual_seed(3)) * 0.02).to(torch.bfloat16)
        for t in (1, 2):
            emb.step_sparse(W, i, r, 1e-3, t)
        outs.append((W, emb.state.clone(), emb.device_status()))
    assert outs[0][2] == 0 and outs[1][2] == EMBER_ERR_ID_OUT_OF_RANGE
    assert torch.equal(outs[0][0].view(torch.int16), outs[1][0].view(torch.int16))
    assert torch.equal(outs[0][1].view(torch.int32), outs[1][1].view(torch.int32))


def test_sparse_v1_and_tiny(cuda_device):
    opt = Opt()
    for V, D, N in [(1, 1, 5), (1, 4, 1), (2, 3, 9)]:
        emb = make(V, D, "f32", N)
        W = torch.randn(V, D, device=cuda_device)
        for t in range(1, 3):
            ids = torch.randint(0, V, (N,), device=cuda_device)
            rows = torch.randn(N, D, device=cuda_device) * 1e-3
            gated_sparse_step(emb, W, ids, rows, 1e-3, t, opt)


def test_sparse_deterministic(cuda_device):
    V, D, N = 50000, 1024, 30000
    outs = []
    for _ in range(2):
        emb = make(V, D, "bf16", N)
        W = (torch.randn(V, D, device=cuda_device, generator=torch.Generator(device=cuda_device)
                         .manual_seed(1)) * 0.02).to(torch.bfloat16)
        for t in range(1, 4):
            ids, rows = batch(V, D, N, t, cuda_device, seed=2)
            emb.step_sparse(W, ids, rows, 1e-3, t)
        outs.append((W.clone(), emb.state.clone()))
    assert torch.equal(outs[0][0].view(torch.int16), outs[1][0].view(torch.int16))
    assert torch.equal(outs[0][1], outs[1][1])


def test_sparse_workload_262144x2048(cuda_device):
    """The sparse embedding workload: 8 x 4096 Zipf(1.1) ids per step over
    V = 262144, D = 2048, bf16 weights; gated steps 1, 2, 3 and 100."""
    wl = synth.WORKLOADS["sparse_v262144_d2048_bf16_n32768"]
    emb = make(wl.V, wl.D, wl.wdtype, wl.N)
    W = synth.init_weights(wl, 0, cuda_device)
    for t in range(1, wl.steps + 1):
        ids, rows = synth.sparse_batch(wl, 0, t, cuda_device)
        if t in (1, 2, 3, wl.steps):
            gated_sparse_step(emb, W, ids, rows, wl.lr, t, Opt())
            if t == 1:
                check_dedup(emb, ids)
        else:
            emb.step_sparse(W, ids, rows, wl.lr, t)
    assert emb.device_status() == 0


def test_sparse_graph_capture_matches_eager(cuda_device):
    """A sparse step is a fixed sequence of launches for a given N, so it can be
    captured in a CUDA graph; replaying it gives the eager result bit for bit."""
    V, D, N = 20000, 512, 9000
    e1, e2 = make(V, D, "bf16", N), make(V, D, "bf16", N)
    W0 = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    W1, W2 = W0.clone(), W0.clone()
    ids, rows = batch(V, D, N, 1, cuda_device, seed=4)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        e2.step_sparse(W2, ids, rows, 1e-3, 1, stream=s)  # warm-up outside the capture
    torch.cuda.synchronize()
    W2.copy_(W0)
    e2.state.zero_()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        e2.step_sparse(W2, ids, rows, 1e-3, 1, stream=s)
    graph.replay()
    e1.step_sparse(W1, ids, rows, 1e-3, 1)
    torch.cuda.synchronize()
    assert torch.equal(W1.view(torch.int16), W2.view(torch.int16))
    assert torch.equal(e1.state, e2.state)
