"""Dense Ember step on the GPU against the CPU oracle (Algorithm 1).

Every check goes through the C ABI (paper_2607_01455_gb300.ember).  Each
gated step starts the oracle from the GPU's own W_{t-1} and state_{t-1}, so
one step's rounding is compared at a time; the bar is a relative error of
1e-5 on the fp32 state and fp32 weights and 1 ulp on bf16 weights.
"""
import numpy as np
import pytest
import torch

from paper_2607_01455_gb300 import synth
from paper_2607_01455_gb300.ember import Ember, EmberError
from parity import Opt, gated_dense_step

pytestmark = pytest.mark.gpu


def make(V, D, wdtype, opt=None, **kw):
    opt = opt or Opt()
    return Ember(V, D, wdtype=wdtype, beta2=opt.beta2, eps=opt.eps, maximize=opt.maximize,
                 bias_correction=opt.bias_correction, variant=opt.variant, **kw)


def rand_grad(V, D, t, device, seed=0, zero_rows=()):
    g = torch.Generator(device=device)
    g.manual_seed(seed * 7919 + t)
    G = torch.randn(V, D, generator=g, device=device) * 1e-3
    G *= torch.rand(V, 1, generator=g, device=device) * 2 + 0.01
    if len(zero_rows):
        G[list(zero_rows)] = 0
    return G


def rand_w(V, D, wdtype, device, seed=0):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    W = torch.randn(V, D, generator=g, device=device) * 0.02
    return W.to(torch.bfloat16 if wdtype == "bf16" else torch.float32)


# Shapes that span several CTAs, row groups and a ragged tail: D not a
# multiple of 4 takes the scalar path; V below, at and above the 304-CTA grid.
SHAPES = [
    (1, 1), (1, 4), (2, 3), (7, 5), (37, 64), (303, 96), (304, 128), (305, 132),
    (1000, 200), (1000, 203), (3001, 256), (777, 1028), (2049, 896), (513, 2048),
    (64, 2047), (150, 4096), (40, 8192), (2, 1), (1000, 33), (7, 127),
]


@pytest.mark.parametrize("V,D", SHAPES)
@pytest.mark.parametrize("wdtype", ["bf16", "f32"])
def test_dense_parity_small_shapes(cuda_device, V, D, wdtype):
    opt = Opt()
    emb = make(V, D, wdtype, opt)
    W = rand_w(V, D, wdtype, cuda_device, seed=V + D)
    for t in range(1, 4):
        G = rand_grad(V, D, t, cuda_device, seed=V * 31 + D, zero_rows=[0] if V > 2 else [])
        gated_dense_step(emb, W, G, 1e-3, t, opt)


@pytest.mark.parametrize("opt", [
    Opt(beta2=0.9, eps=1e-6), Opt(maximize=True), Opt(bias_correction=False),
    Opt(variant="row"), Opt(variant="col"), Opt(beta2=0.0), Opt(eps=0.0),
], ids=["beta2_0.9", "maximize", "no_bias_correction", "row_only", "col_only", "beta2_0", "eps_0"])
@pytest.mark.parametrize("V,D", [(1000, 200), (2049, 896)])
def test_dense_parity_hyperparameters(cuda_device, opt, V, D):
    emb = make(V, D, "bf16", opt)
    W = rand_w(V, D, "bf16", cuda_device)
    for t in range(1, 5):
        gated_dense_step(emb, W, rand_grad(V, D, t, cuda_device, seed=3), 2e-3, t, opt)


@pytest.mark.parametrize("V,D,wdtype", [(305, 8192, "bf16"), (1000, 4096, "bf16"), (2049, 896, "bf16"),
                                         (777, 203, "f32"), (3001, 64, "bf16"), (1, 8, "bf16"),
                                         (7, 5, "f32")])
def test_row_only_single_pass_parity(cuda_device, V, D, wdtype):
    """The row-only variant runs as one fused pass over G and W; it must
    still match the oracle's row-only step, state included."""
    opt = Opt(variant="row")
    emb = make(V, D, wdtype, opt)
    W = rand_w(V, D, wdtype, cuda_device, seed=D)
    for t in range(1, 4):
        G = rand_grad(V, D, t, cuda_device, seed=V, zero_rows=[0] if V > 2 else [])
        gated_dense_step(emb, W, G, 1e-3, t, opt)


def test_dense_workload_small_all_steps(cuda_device):
    """The 1024 x 64 fp32 workload, all 10 steps, each gated."""
    wl = synth.WORKLOADS["dense_v1024_d64_f32"]
    emb = make(wl.V, wl.D, wl.wdtype)
    W = synth.init_weights(wl, 0, cuda_device)
    for t in range(1, wl.steps + 1):
        gated_dense_step(emb, W, synth.dense_grad(wl, 0, t, cuda_device), wl.lr, t, Opt())


def _run_workload(cuda_device, name, gate_steps, steps=None):
    wl = synth.WORKLOADS[name]
    emb = make(wl.V, wl.D, wl.wdtype)
    W = synth.init_weights(wl, 0, cuda_device)
    scales = synth.row_scales(wl, cuda_device)
    sets = synth.row_sets(wl, 0)
    G = torch.empty(wl.V, wl.D, device=cuda_device)
    last = steps or wl.steps
    for t in range(1, last + 1):
        synth.dense_grad(wl, 0, t, cuda_device, out=G, scales=scales, sets=sets)
        if t in gate_steps:
            gated_dense_step(emb, W, G, wl.lr, t, Opt(), all_cores=True)
        else:
            emb.step_dense(W, G, wl.lr, t)
    torch.cuda.synchronize()
    return wl, emb, W, sets


def test_dense_workload_32000x4096(cuda_device):
    _run_workload(cuda_device, "dense_v32000_d4096_bf16", {1, 2, 3, 50, 100})


def test_dense_workload_tied_151936x896(cuda_device):
    wl, emb, W, (zero_rows, _) = _run_workload(
        cuda_device, "dense_tied_v151936_d896_bf16", {1, 2, 3, 50, 100})
    # never-seen tokens: r stays exactly zero and their rows never move
    assert torch.all(emb.r[zero_rows.to(cuda_device)] == 0)
    W0 = synth.init_weights(wl, 0, cuda_device)
    zr = zero_rows.to(cuda_device)
    assert torch.equal(W[zr].view(torch.int16), W0[zr].view(torch.int16))


def test_dense_workload_lmhead_128256x8192(cuda_device):
    """The large LM head in the launch configuration the benchmark times,
    gated at steps 1, 2, 3, 10, 20, 30, 40 and 50."""
    _run_workload(cuda_device, "dense_lmhead_v128256_d8192_bf16", {1, 2, 3, 10, 20, 30, 40, 50})


def test_dense_deterministic_and_resumable(cuda_device):
    """Bit-identical on a rerun (Section 2.3), and a run restored from a saved
    (W, state) after step 4 continues exactly like the uninterrupted one."""
    V, D = 3001, 1024
    runs = []
    for _ in range(2):
        emb = make(V, D, "bf16")
        W = rand_w(V, D, "bf16", cuda_device)
        for t in range(1, 8):
            emb.step_dense(W, rand_grad(V, D, t, cuda_device), 1e-3, t)
            if t == 4:
                saved = (W.clone(), emb.state.clone())
        runs.append((W.clone(), emb.state.clone()))
    assert torch.equal(runs[0][0].view(torch.int16), runs[1][0].view(torch.int16))
    assert torch.equal(runs[0][1], runs[1][1])
    emb = make(V, D, "bf16")
    W, st = saved
    emb.state.copy_(st)
    for t in range(5, 8):
        emb.step_dense(W, rand_grad(V, D, t, cuda_device), 1e-3, t)
    assert torch.equal(W.view(torch.int16), runs[0][0].view(torch.int16))
    assert torch.equal(emb.state, runs[0][1])


@pytest.mark.parametrize("m", [6, -7])
def test_dense_power_of_two_scale_invariance(cuda_device, m):
    """eps = 0: G and 2^m G give bit-identical weights (the update is a
    z-score, appendix 'Outer Product Unit Alignment')."""
    V, D = 1000, 512
    a, b = make(V, D, "bf16", Opt(eps=0.0)), make(V, D, "bf16", Opt(eps=0.0))
    Wa, Wb = rand_w(V, D, "bf16", cuda_device), rand_w(V, D, "bf16", cuda_device)
    for t in range(1, 4):
        G = rand_grad(V, D, t, cuda_device)
        a.step_dense(Wa, G, 1e-3, t)
        b.step_dense(Wb, G * 2.0 ** m, 1e-3, t)
    assert torch.equal(Wa.view(torch.int16), Wb.view(torch.int16))
    assert torch.equal(a.r * 2.0 ** (2 * m), b.r)


def test_dense_all_zero_gradient_is_a_no_op(cuda_device):
    V, D = 500, 256
    emb = make(V, D, "bf16")
    W = rand_w(V, D, "bf16", cuda_device)
    W0 = W.clone()
    emb.step_dense(W, torch.zeros(V, D, device=cuda_device), 1e-3, 1)
    assert torch.equal(W.view(torch.int16), W0.view(torch.int16))
    assert torch.all(emb.state == 0)
    assert emb.device_status() == 0


def test_dense_misaligned_pointers_take_the_scalar_path(cuda_device):
    """Views one element into a buffer are not 16-byte aligned; the step still
    matches the oracle.  (Wide misaligned rows run in scalar column panels:
    test_wide_gpu.py.)"""
    V, D = 300, 128
    opt = Opt()
    emb = make(V, D, "bf16", opt)
    Wbuf = rand_w(V * D + 1, 1, "bf16", cuda_device).view(-1)
    W = Wbuf[1:].view(V, D)
    Gbuf = torch.randn(V * D + 1, device=cuda_device) * 1e-3
    G = Gbuf[1:].view(V, D)
    for t in range(1, 3):
        gated_dense_step(emb, W, G, 1e-3, t, opt)


def test_dense_graph_capture_matches_eager(cuda_device):
    """The step is a fixed sequence of launches on the caller's stream, so it
    can be captured in a CUDA graph; the replay gives the eager result."""
    V, D = 2049, 896
    e1, e2 = make(V, D, "bf16"), make(V, D, "bf16")
    W1, W2 = rand_w(V, D, "bf16", cuda_device), rand_w(V, D, "bf16", cuda_device)
    G = rand_grad(V, D, 1, cuda_device)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        e2.step_dense(W2, G, 1e-3, 1, stream=s)  # warm-up on the side stream
        W2.copy_(rand_w(V, D, "bf16", cuda_device))
        e2.state.zero_()
    torch.cuda.synchronize()
    with torch.cuda.graph(graph, stream=s):
        e2.step_dense(W2, G, 1e-3, 1, stream=s)
    graph.replay()
    e1.step_dense(W1, G, 1e-3, 1)
    torch.cuda.synchronize()
    assert torch.equal(W1.view(torch.int16), W2.view(torch.int16))
    assert torch.equal(e1.state, e2.state)


@pytest.mark.parametrize("V,D,wdtype", [(3001, 1024, "bf16"), (2000, 8192, "bf16"), (513, 203, "f32")])
def test_step_from_host_matches_device_step(cuda_device, V, D, wdtype):
    """The gradient read from pinned host memory (and staged in HBM by the
    reduce pass) gives the same W and state, bit for bit, as the step on a
    device-resident gradient; the stage holds an exact copy of G."""
    a, b = make(V, D, wdtype), make(V, D, wdtype)
    Wa = rand_w(V, D, wdtype, cuda_device)
    Wb = Wa.clone()
    stage = torch.empty(V, D, device=cuda_device)
    for t in (1, 2):
        G = rand_grad(V, D, t, cuda_device, seed=D)
        Gh = G.cpu().pin_memory()
        a.step_dense(Wa, G, 1e-3, t)
        b.step_dense_from_host(Wb, Gh, stage, 1e-3, t)
        torch.cuda.synchronize()
        assert torch.equal(stage, G)
        assert torch.equal(Wa.view(torch.int16) if wdtype == "bf16" else Wa,
                           Wb.view(torch.int16) if wdtype == "bf16" else Wb)
        assert torch.equal(a.state, b.state)


def test_step_from_host_refuses_unregistered_memory(cuda_device):
    V, D = 64, 32
    emb = make(V, D, "bf16")
    W = rand_w(V, D, "bf16", cuda_device)
    pageable = np.zeros((V, D), np.float32)
    stage = torch.empty(V, D, device=cuda_device)
    with pytest.raises(EmberError) as ex:
        emb.step_dense_from_host(W, pageable.ctypes.data, stage, 1e-3, 1)
    assert ex.value.status == 1  # EMBER_ERR_INVALID_ARG


@pytest.mark.parametrize("V,D,wdtype", [(1024, 64, "f32"), (256, 256, "bf16"), (100, 300, "f32"), (1, 4, "bf16"),
                                         (305, 132, "bf16"), (7, 12, "f32"), (2048, 32, "bf16"),
                                         (3001, 1024, "bf16"), (40, 8192, "bf16")])
def test_one_launch_and_three_launch_forms_agree_bitwise(cuda_device, V, D, wdtype):
    """A small table runs as one cluster launch (G and W kept in shared
    memory, the column statistics exchanged through distributed shared
    memory) and, while trace events are set, as three launches (reduce,
    state, apply).  Both run the same arithmetic on the same CTA row ranges,
    with the column totals summed exactly, so they give the same bits (the
    last two shapes take three launches either way)."""
    a, b = make(V, D, wdtype), make(V, D, wdtype)
    Wa = rand_w(V, D, wdtype, cuda_device, seed=5)
    Wb = Wa.clone()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    b.trace(ev)
    for t in range(1, 5):
        G = rand_grad(V, D, t, cuda_device, seed=D)
        a.step_dense(Wa, G, 1e-3, t)
        b.step_dense(Wb, G, 1e-3, t)
    torch.cuda.synchronize()
    b.trace([])
    view = torch.int16 if wdtype == "bf16" else torch.int32
    assert torch.equal(Wa.view(view), Wb.view(view))
    assert torch.equal(a.state.view(torch.int32), b.state.view(torch.int32))
    assert a.device_status() == 0 and b.device_status() == 0
