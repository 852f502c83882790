"""LM-head gradient on the tensor cores and the Ember step fused with it,
against the CPU oracle.

G = dlogits^T H is the sum over T tokens of the outer product of each
token's softmax error and hidden state (appendix "Decomposing the Squared
Gradient").  The kernel multiplies bf16 factors (exact in fp32) and
accumulates in fp32 in an order of its own; the oracle sums the same
products in fp64 in token order.  Bound used here, for any summation order
of T exactly representable terms with an fp32 accumulator that may truncate
instead of round: |G - G_exact| <= (T + 1) 2^-22 sum_t |delta h| (one
2-ulp error per addition, plus the final rounding), with the oracle's own
fp64 error far below it.

The fused step is then checked like the dense step: from the GPU's own
W_{t-1} and state_{t-1}, the oracle's step on the G the GPU formed must give
W_t and the state within 1e-5 relative (1 ulp for bf16 weights).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01455_gb300 import synth
from paper_2607_01455_gb300.ember import Ember
from parity import Opt, check_state, check_weights, oracle_kwargs, w_to_host

pytestmark = pytest.mark.gpu


def bits(x):
    return x.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def check_gemm(G, dl, h, rows=None):
    """G (device, fp32) against the oracle's fp64 G = dl^T h within the bound."""
    T = dl.shape[0]
    G64, A64 = oracle.lmhead_grad(bits(dl), bits(h), rows=rows)
    Gg = G.detach().cpu().numpy().astype(np.float64)
    if rows is not None:
        Gg = Gg[rows]
    err = np.abs(Gg - G64)
    bound = (T + 1) * 2.0 ** -22 * A64 + 2.0 ** -126
    ratio = err / bound
    k = np.unravel_index(int(ratio.argmax()), ratio.shape)
    assert ratio[k] <= 1.0, f"G{k}: {Gg[k]!r} vs {G64[k]!r}, {ratio[k]:.3g} of the bound"
    return float(ratio.max())


def make(V, D, wdtype="bf16", opt=None):
    opt = opt or Opt()
    return Ember(V, D, wdtype=wdtype, beta2=opt.beta2, eps=opt.eps, maximize=opt.maximize,
                 bias_correction=opt.bias_correction, variant=opt.variant)


# (V, D, T): one tile, partial tiles in every direction (V not a multiple of
# 128, D not of 256, T not of 64), several tiles per CTA, the widest D.
SHAPES = [
    (8, 8, 1), (128, 256, 64), (136, 264, 65), (1000, 328, 100), (384, 512, 192),
    (2048, 1024, 300), (1024, 8192, 64), (4096, 256, 17), (19520, 512, 129),
]


@pytest.mark.parametrize("V,D,T", SHAPES)
def test_lmhead_grad_matches_oracle(cuda_device, V, D, T):
    emb = make(V, D)
    dl, h = synth.lmhead_inputs(V, D, T, seed=V + D + T, t=1, device=cuda_device)
    G = torch.full((V, D), float("nan"), device=cuda_device)
    emb.lmhead_grad(dl, h, G)
    assert emb.device_status() == 0
    rows = None if V * D * T <= 2 ** 28 else np.unique(np.r_[0:64, V - 64:V, np.arange(0, V, 97)])
    check_gemm(G, dl, h, rows)


def test_lmhead_grad_one_hot_errors_gather_hidden_rows_exactly(cuda_device):
    """delta_t = -e_{y_t} and small-integer hidden states: every partial sum
    is an integer below 2^24, so G must equal the gathered sums exactly."""
    V, D, T = 1000, 264, 300
    g = torch.Generator(device="cpu").manual_seed(5)
    y = torch.randint(0, V - 8, (T,), generator=g)
    dl = torch.zeros(T, V, dtype=torch.bfloat16)
    dl[torch.arange(T), y] = -1.0
    h = torch.randint(-8, 9, (T, D), generator=g).to(torch.bfloat16)
    want = np.zeros((V, D))
    np.add.at(want, y.numpy(), -h.float().numpy().astype(np.float64))
    emb = make(V, D)
    G = torch.full((V, D), float("nan"), device=cuda_device)
    emb.lmhead_grad(dl.to(cuda_device), h.to(cuda_device), G)
    np.testing.assert_array_equal(G.cpu().numpy().astype(np.float64), want)


@pytest.mark.parametrize("V,D,T", [(136, 264, 65), (1000, 328, 100), (2048, 1024, 300), (304, 8192, 40)])
@pytest.mark.parametrize("wdtype", ["bf16", "f32"])
def test_step_lmhead_gated(cuda_device, V, D, T, wdtype):
    opt = Opt()
    emb = make(V, D, wdtype, opt)
    gw = torch.Generator(device=cuda_device).manual_seed(V)
    W = (torch.randn(V, D, generator=gw, device=cuda_device) * 0.02).to(
        torch.bfloat16 if wdtype == "bf16" else torch.float32)
    G = torch.empty(V, D, device=cuda_device)
    for t in range(1, 4):
        dl, h = synth.lmhead_inputs(V, D, T, seed=V + D, t=t, device=cuda_device)
        W0 = w_to_host(W)
        st0 = emb.state.cpu().numpy().copy()
        emb.step_lmhead(W, dl, h, G, 1e-3, t)
        torch.cuda.synchronize()
        assert emb.device_status() == 0
        if t == 1:
            check_gemm(G, dl, h)
        r, c = st0[:V].copy(), st0[V:].copy()
        Wo = W0.copy()
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, float(np.float32(1e-3)), t, **oracle_kwargs(opt))
        st = emb.state.cpu().numpy()
        check_state(st[:V], r, "r")
        check_state(st[V:], c, "c")
        check_weights(w_to_host(W), Wo, 1e-3, prev=W0, record=True)


@pytest.mark.parametrize("opt", [Opt(variant="row"), Opt(variant="col"), Opt(maximize=True),
                                 Opt(bias_correction=False), Opt(beta2=0.9, eps=1e-6)],
                         ids=["row", "col", "maximize", "no-bias-correction", "beta2-0.9"])
def test_step_lmhead_hyperparameters(cuda_device, opt):
    V, D, T = 1000, 328, 100
    emb = make(V, D, "bf16", opt)
    W = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    G = torch.empty(V, D, device=cuda_device)
    for t in (1, 2):
        dl, h = synth.lmhead_inputs(V, D, T, seed=3, t=t, device=cuda_device)
        W0 = w_to_host(W)
        st0 = emb.state.cpu().numpy().copy()
        emb.step_lmhead(W, dl, h, G, 1e-3, t)
        torch.cuda.synchronize()
        r, c = st0[:V].copy(), st0[V:].copy()
        Wo = W0.copy()
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, float(np.float32(1e-3)), t, **oracle_kwargs(opt))
        st = emb.state.cpu().numpy()
        check_state(st[:V], r, "r")
        check_state(st[V:], c, "c")
        check_weights(w_to_host(W), Wo, 1e-3, prev=W0, record=True)


def test_step_lmhead_writes_the_same_G_and_is_deterministic(cuda_device):
    V, D, T = 2048, 1024, 300
    dl, h = synth.lmhead_inputs(V, D, T, seed=9, t=1, device=cuda_device)
    runs = []
    for _ in range(2):
        emb = make(V, D)
        W = (torch.randn(V, D, device=cuda_device, generator=torch.Generator(device=cuda_device).manual_seed(1))
             * 0.02).to(torch.bfloat16)
        G = torch.empty(V, D, device=cuda_device)
        emb.step_lmhead(W, dl, h, G, 1e-3, 1)
        G2 = torch.empty(V, D, device=cuda_device)
        emb.lmhead_grad(dl, h, G2)
        torch.cuda.synchronize()
        assert torch.equal(G.view(torch.int32), G2.view(torch.int32))
        runs.append((W.view(torch.int16).clone(), emb.state.view(torch.int32).clone(), G))
    assert torch.equal(runs[0][0], runs[1][0])
    assert torch.equal(runs[0][1], runs[1][1])
    assert torch.equal(runs[0][2].view(torch.int32), runs[1][2].view(torch.int32))


def test_step_lmhead_equals_dense_step_on_its_gradient(cuda_device):
    """The fused step and ember_step_dense on the same G, from the same W and
    state, agree to rounding: only the grouping of the sums of g^2 differs."""
    V, D, T = 4096, 2048, 256
    a, b = make(V, D), make(V, D)
    W = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    G = torch.empty(V, D, device=cuda_device)
    for t in range(1, 4):  # build up a state
        dl, h = synth.lmhead_inputs(V, D, T, seed=4, t=t, device=cuda_device)
        a.step_lmhead(W, dl, h, G, 1e-3, t)
    b.state.copy_(a.state)
    Wb = W.clone()
    dl, h = synth.lmhead_inputs(V, D, T, seed=4, t=4, device=cuda_device)
    a.step_lmhead(W, dl, h, G, 1e-3, 4)
    b.step_dense(Wb, G, 1e-3, 4)
    torch.cuda.synchronize()
    check_state(a.state.cpu().numpy(), b.state.cpu().numpy(), "state")
    check_weights(w_to_host(W), w_to_host(Wb), 1e-3)


def test_lmhead_full_size_sampled(cuda_device):
    """The 128256 x 8192, T = 4096 LM head: G on sampled rows against the
    oracle (the most frequent targets, the first and last rows, a stride),
    and the fused step against ember_step_dense on the same G."""
    wl = synth.WORKLOADS["lmhead_grad_v128256_d8192_t4096_bf16"]
    V, D, T = wl.V, wl.D, wl.T
    a = make(V, D)
    b = make(V, D)
    W = synth.init_weights(wl, 0, cuda_device)
    G = torch.empty(V, D, device=cuda_device)
    dl, h = synth.lmhead_inputs(V, D, T, seed=0, t=1, device=cuda_device)
    Wb = W.clone()
    a.step_lmhead(W, dl, h, G, wl.lr, 1)
    b.step_dense(Wb, G, wl.lr, 1)
    torch.cuda.synchronize()
    assert a.device_status() == 0
    rows = np.unique(np.r_[0:6, 100, 1000, 77777, V - 1, np.arange(17, V, V // 6)])
    check_gemm(G, dl, h, rows)
    check_state(b.state.cpu().numpy(), a.state.cpu().numpy(), "state")
    # bf16 W, compared on the GPU (2 GB per copy): within 1 ulp, or, where
    # the new weight nearly cancels, within 1e-5 of max(|W|, lr)
    def ordinal(x):
        i = x.view(torch.int16).to(torch.int32)
        return torch.where(i < 0, -(i & 0x7FFF), i)
    d = (ordinal(W) - ordinal(Wb)).abs()
    far = d > 1
    assert int(far.sum()) <= 1e-3 * d.numel()
    if bool(far.any()):
        wa, wb = W[far].double(), Wb[far].double()
        assert float(((wa - wb).abs() / wb.abs().clamp(min=wl.lr)).max()) <= 1e-5


def test_step_lmhead_graph_capture_matches_eager(cuda_device):
    """The fused step (cluster launch of the tensor-core kernel, state, apply)
    is a fixed sequence of launches, so a CUDA graph of it replays to the
    eager result, bit for bit, and keeps stepping correctly."""
    V, D, T = 2048, 1024, 300
    e1, e2 = make(V, D), make(V, D)
    W0 = (torch.randn(V, D, device=cuda_device) * 0.02).to(torch.bfloat16)
    W1, W2 = W0.clone(), W0.clone()
    G1, G2 = torch.empty(V, D, device=cuda_device), torch.empty(V, D, device=cuda_device)
    dl, h = synth.lmhead_inputs(V, D, T, seed=6, t=1, device=cuda_device)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        e2.step_lmhead(W2, dl, h, G2, 1e-3, 1, stream=s)  # warm-up on the side stream
        W2.copy_(W0)
        e2.state.zero_()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        e2.step_lmhead(W2, dl, h, G2, 1e-3, 1, stream=s)
    for _ in range(2):  # two replays = two steps at t = 1 (the t is baked into the graph)
        graph.replay()
        e1.step_lmhead(W1, dl, h, G1, 1e-3, 1)
    torch.cuda.synchronize()
    assert e2.device_status() == 0
    assert torch.equal(G1.view(torch.int32), G2.view(torch.int32))
    assert torch.equal(W1.view(torch.int16), W2.view(torch.int16))
    assert torch.equal(e1.state.view(torch.int32), e2.state.view(torch.int32))


def test_bounded_wait_gives_up_and_the_next_step_recovers(cuda_device):
    """The LM-head kernel's main-loop mbarrier waits, made 1 ns long, give up
    for real: the kernel stops every role, lets the copies and MMAs it has
    issued complete (its teardown waits keep their 2 s limit), frees its
    tensor memory and returns, and the sticky flag reads EMBER_ERR_TIMEOUT.
    The context stays usable: back at the default limit, the fused step on
    the same handle passes the oracle gate."""
    from paper_2607_01455_gb300.ember import EMBER_ERR_TIMEOUT
    V, D, T = 2048, 1024, 4096  # 64 pipeline stages per tile: many waits
    emb = make(V, D, "f32")
    dl, h = synth.lmhead_inputs(V, D, T, seed=9, t=1, device=cuda_device)
    G = torch.zeros(V, D, device=cuda_device)
    emb.set_wait_limit_ns(1)
    emb.lmhead_grad(dl, h, G)
    assert emb.device_status() == EMBER_ERR_TIMEOUT
    assert emb.device_status() == 0  # read and cleared
    emb.set_wait_limit_ns(0)
    gw = torch.Generator(device=cuda_device).manual_seed(4)
    W = torch.randn(V, D, generator=gw, device=cuda_device) * 0.02
    for t in (1, 2):
        dl, h = synth.lmhead_inputs(V, D, T, seed=9, t=t, device=cuda_device)
        W0 = w_to_host(W)
        st0 = emb.state.cpu().numpy().copy()
        emb.step_lmhead(W, dl, h, G, 1e-3, t)
        torch.cuda.synchronize()
        assert emb.device_status() == 0
        if t == 1:
            check_gemm(G, dl, h, rows=np.arange(0, V, 7))
        r, c = st0[:V].copy(), st0[V:].copy()
        Wo = W0.copy()
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, float(np.float32(1e-3)), t)
        st = emb.state.cpu().numpy()
        check_state(st[:V], r, "r")
        check_state(st[V:], c, "c")
        check_weights(w_to_host(W), Wo, 1e-3, prev=W0, record=True)
