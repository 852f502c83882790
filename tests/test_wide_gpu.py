"""Tables whose rows a CTA cannot hold whole: D > 8192 on the 16-byte vector
path, D > 2048 on the scalar one.  They run in equal column panels (one
reduce and one apply launch per panel; each row's sum of g^2 is added up
from per-panel partial sums), and every result must still match the oracle
of Algorithm 1, which knows nothing of panels.

Panel splits covered: 2, 3 and 8 panels of 8192 columns; 2 panels of 4100
and of 6144; scalar panels (D not a multiple of 4) of 1501, 2001 and, at
the widest table accepted but one, 32 of 2048 with a narrower last one; and
a misaligned view of a 4096-wide table (scalar path, 2 panels of 2048).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01455_gb300 import ember as E
from paper_2607_01455_gb300 import synth
from paper_2607_01455_gb300.ember import Ember, EmberError
from parity import Opt, check_state, check_weights, gated_dense_step, oracle_kwargs, w_to_host

pytestmark = pytest.mark.gpu


def make(V, D, wdtype, opt=None, **kw):
    opt = opt or Opt()
    return Ember(V, D, wdtype=wdtype, beta2=opt.beta2, eps=opt.eps, maximize=opt.maximize,
                 bias_correction=opt.bias_correction, variant=opt.variant, **kw)


def rand_w(V, D, wdtype, device, seed=0):
    g = torch.Generator(device=device).manual_seed(seed)
    W = torch.randn(V, D, generator=g, device=device) * 0.02
    return W.to(torch.bfloat16 if wdtype == "bf16" else torch.float32)


def rand_grad(V, D, t, device, seed=0):
    g = torch.Generator(device=device).manual_seed(seed * 7919 + t)
    G = torch.randn(V, D, generator=g, device=device) * 1e-3
    G *= torch.rand(V, 1, generator=g, device=device) * 2 + 0.01
    if V > 2:
        G[1] = 0  # a row with no gradient keeps r decaying and W unchanged
    # column energy that differs by panel, so a panel's statistics cannot
    # stand in for another's
    G *= torch.linspace(0.5, 2.0, D, device=device)
    return G


def bits(x):
    return x.view(torch.int16) if x.dtype == torch.bfloat16 else x.view(torch.int32)


WIDE = [(300, 8196, "bf16"), (129, 16384, "f32"), (257, 12288, "bf16"), (64, 24576, "bf16"),
        (33, 65536, "bf16"), (100, 3001, "bf16"), (50, 10001, "f32"), (305, 8200, "f32"),
        (9, 65533, "f32")]


@pytest.mark.parametrize("V,D,wdtype", WIDE)
def test_wide_dense_parity(cuda_device, V, D, wdtype):
    opt = Opt()
    emb = make(V, D, wdtype, opt)
    W = rand_w(V, D, wdtype, cuda_device, seed=D)
    for t in range(1, 4):
        gated_dense_step(emb, W, rand_grad(V, D, t, cuda_device, seed=V), 1e-3, t, opt)
    assert emb.device_status() == 0


@pytest.mark.parametrize("opt", [Opt(variant="row"), Opt(variant="col"), Opt(maximize=True),
                                 Opt(bias_correction=False), Opt(beta2=0.9, eps=1e-6)],
                         ids=["row", "col", "maximize", "no-bias-correction", "beta2-0.9"])
def test_wide_dense_hyperparameters(cuda_device, opt):
    """The row-only variant has no one-pass kernel for panels; it runs the
    three passes with a unit column scale."""
    V, D = 300, 12288
    emb = make(V, D, "bf16", opt)
    W = rand_w(V, D, "bf16", cuda_device, seed=1)
    for t in range(1, 4):
        gated_dense_step(emb, W, rand_grad(V, D, t, cuda_device, seed=2), 2e-3, t, opt)


def test_wide_misaligned_view_takes_scalar_panels(cuda_device):
    """A view one element into its buffer is not 16-byte aligned: the scalar
    path holds 2048 columns per CTA, so D = 4096 runs as two panels."""
    V, D = 200, 4096
    opt = Opt()
    emb = make(V, D, "bf16", opt)
    W = rand_w(V * D + 1, 1, "bf16", cuda_device, seed=3).view(-1)[1:].view(V, D)
    Gbuf = torch.empty(V * D + 1, device=cuda_device)
    for t in range(1, 3):
        G = Gbuf[1:].view(V, D)
        G.copy_(rand_grad(V, D, t, cuda_device, seed=4))
        gated_dense_step(emb, W, G, 1e-3, t, opt)


def test_wide_dense_deterministic_and_graph_capture(cuda_device):
    V, D = 1000, 16384
    e1, e2 = make(V, D, "bf16"), make(V, D, "bf16")
    W1 = rand_w(V, D, "bf16", cuda_device, seed=5)
    W2 = W1.clone()
    G = rand_grad(V, D, 1, cuda_device, seed=6)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        e2.step_dense(W2, G, 1e-3, 1, stream=s)  # warm-up on the side stream
    torch.cuda.synchronize()
    W2.copy_(W1)
    e2.state.zero_()
    with torch.cuda.graph(graph, stream=s):
        e2.step_dense(W2, G, 1e-3, 1, stream=s)
    graph.replay()
    e1.step_dense(W1, G, 1e-3, 1)
    torch.cuda.synchronize()
    assert torch.equal(bits(W1), bits(W2))
    assert torch.equal(e1.state, e2.state)


def test_wide_from_host_matches_device_step(cuda_device):
    V, D = 513, 16384
    a, b = make(V, D, "bf16"), make(V, D, "bf16")
    Wa = rand_w(V, D, "bf16", cuda_device, seed=7)
    Wb = Wa.clone()
    stage = torch.empty(V, D, device=cuda_device)
    for t in (1, 2):
        G = rand_grad(V, D, t, cuda_device, seed=8)
        Gh = G.cpu().pin_memory()
        a.step_dense(Wa, G, 1e-3, t)
        b.step_dense_from_host(Wb, Gh, stage, 1e-3, t)
        torch.cuda.synchronize()
        assert torch.equal(stage, G)
        assert torch.equal(bits(Wa), bits(Wb))
        assert torch.equal(a.state, b.state)


@pytest.mark.parametrize("V,D,N", [(2000, 16384, 3000), (2000, 10001, 1500)])
def test_wide_sparse_parity(cuda_device, V, D, N):
    opt = Opt()
    emb = make(V, D, "bf16", opt, max_sparse_N=N)
    W = rand_w(V, D, "bf16", cuda_device, seed=9)
    p = (torch.arange(V, device=cuda_device, dtype=torch.float64) + 1) ** -1.1
    cdf = torch.cumsum(p, 0)
    cdf /= cdf[-1].clone()
    for t in range(1, 4):
        g = torch.Generator(device=cuda_device).manual_seed(10 + t)
        u = torch.rand(N, generator=g, device=cuda_device, dtype=torch.float64)
        ids = torch.searchsorted(cdf, u, right=True).clamp_(max=V - 1).to(torch.int64)
        rows = torch.randn(N, D, generator=g, device=cuda_device) * 1e-4
        W0 = w_to_host(W)
        st0 = emb.state.cpu().numpy().copy()
        emb.step_sparse(W, ids, rows, 1e-3, t)
        torch.cuda.synchronize()
        assert emb.device_status() == 0
        r, c = st0[:V].copy(), st0[V:].copy()
        Wo = W0.copy()
        oracle.step_sparse(Wo, ids.cpu().numpy(), rows.cpu().numpy(), r, c, float(np.float32(1e-3)), t,
                           **oracle_kwargs(opt))
        st = emb.state.cpu().numpy()
        check_state(st[:V], r, "r")
        check_state(st[V:], c, "c")
        Wg = w_to_host(W)
        check_weights(Wg, Wo, 1e-3, prev=W0, record=True, summed_input=True)
        touched = np.zeros(V, bool)
        touched[ids.cpu().numpy()] = True
        assert np.array_equal(Wg[~touched], W0[~touched])


@pytest.mark.parametrize("V,D,T", [(1000, 8200, 64), (264, 16384, 40)])
def test_wide_step_lmhead_gated(cuda_device, V, D, T):
    opt = Opt()
    emb = make(V, D, "bf16", opt)
    W = rand_w(V, D, "bf16", cuda_device, seed=11)
    G = torch.empty(V, D, device=cuda_device)
    for t in range(1, 3):
        dl, h = synth.lmhead_inputs(V, D, T, seed=V + D, t=t, device=cuda_device)
        W0 = w_to_host(W)
        st0 = emb.state.cpu().numpy().copy()
        emb.step_lmhead(W, dl, h, G, 1e-3, t)
        torch.cuda.synchronize()
        assert emb.device_status() == 0
        if t == 1:
            # the fp32-accumulation bound of the LM-head tests
            want, absG = oracle.lmhead_grad(dl.cpu().view(torch.int16).numpy().view(np.uint16),
                                            h.cpu().view(torch.int16).numpy().view(np.uint16))
            err = np.abs(G.cpu().numpy().astype(np.float64) - want)
            assert np.all(err <= (T + 1) * 2.0 ** -22 * absG + 2.0 ** -126)
        r, c = st0[:V].copy(), st0[V:].copy()
        Wo = W0.copy()
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, float(np.float32(1e-3)), t, **oracle_kwargs(opt))
        st = emb.state.cpu().numpy()
        check_state(st[:V], r, "r")
        check_state(st[V:], c, "c")
        check_weights(w_to_host(W), Wo, 1e-3, prev=W0, record=True)


def test_wide_tables_are_refused_by_shards_and_noalloc(cuda_device):
    V, D = 64, 16384
    emb = make(V, D, "bf16")
    blk = torch.zeros(emb.shard_scale_bytes(), dtype=torch.uint8, device=cuda_device)
    with pytest.raises(EmberError) as ex:
        emb.shard_reduce(0, 2, torch.zeros(V // 2, D, device=cuda_device), blk)
    assert ex.value.status == E.EMBER_ERR_UNSUPPORTED
    h = E.ember_create(V, D, E.ember_hparams_default(), E.EMBER_BF16)
    try:
        state = torch.zeros(V + D, device=cuda_device)
        W = torch.zeros(V, D, dtype=torch.bfloat16, device=cuda_device)
        with pytest.raises(EmberError) as ex:
            E.ember_step_dense_noalloc(h, W, torch.zeros(V, D, device=cuda_device), state, 1e-3, 1)
        assert ex.value.status == E.EMBER_ERR_WORKSPACE
    finally:
        E.ember_destroy(h)
