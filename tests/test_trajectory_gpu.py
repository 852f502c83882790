"""Ungated trajectories: the GPU and the CPU oracle each run every step of a
workload on their own (no per-step gating), and the drift between the two
at the end is measured and bounded.

Why the drift stays small: the update of W does not depend on W (Algorithm
1), and r, c are exponential averages, which carry an earlier difference
forward scaled by beta2 and never amplify it.  So a difference in W is the
sum of the per-step differences of the increments, each within the gated
bar.  Bounds used (K steps):
  fp32 W:   |W_gpu - W_oracle| <= K * 1e-5 * max(|W|, lr)
  bf16 W:   at most K ulps (one rounding that may land the other way per
            step), and more than 1 ulp on at most 1 % of the elements
  r, c:     relative 1e-5, exact zeros stay exact
The measured drift is printed (pytest -s).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01455_gb300 import synth
from paper_2607_01455_gb300.ember import Ember
from parity import bf16_ulp_distance, check_state, w_to_host

pytestmark = pytest.mark.gpu


def report(name, **kw):
    print(f"\n[trajectory] {name}: " + ", ".join(f"{k}={v}" for k, v in kw.items()))


def test_dense_fp32_trajectory_all_steps(cuda_device):
    wl = synth.WORKLOADS["dense_v1024_d64_f32"]
    emb = Ember(wl.V, wl.D, wdtype=wl.wdtype, device=cuda_device)
    W = synth.init_weights(wl, 0, cuda_device)
    Wo = w_to_host(W)
    r, c = np.zeros(wl.V, np.float32), np.zeros(wl.D, np.float32)
    lr32 = float(np.float32(wl.lr))
    for t in range(1, wl.steps + 1):
        G = synth.dense_grad(wl, 0, t, cuda_device)
        emb.step_dense(W, G, wl.lr, t)
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, lr32, t)
    torch.cuda.synchronize()
    st = emb.state.cpu().numpy()
    check_state(st[:wl.V], r, "r")
    check_state(st[wl.V:], c, "c")
    Wg = w_to_host(W).astype(np.float64)
    rel = np.abs(Wg - Wo) / np.maximum(np.abs(Wo), wl.lr)
    report(wl.name, steps=wl.steps, max_rel_W=f"{rel.max():.3g}")
    assert rel.max() <= wl.steps * 1e-5


@pytest.mark.parametrize("V,D,steps", [(2000, 512, 20), (777, 1028, 10)])
def test_dense_bf16_trajectory(cuda_device, V, D, steps):
    wl = synth.Workload(f"dense_v{V}_d{D}_bf16", V, D, "bf16", steps)
    emb = Ember(V, D, wdtype="bf16", device=cuda_device)
    W = synth.init_weights(wl, 1, cuda_device)
    Wo = w_to_host(W)
    r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
    scales = synth.row_scales(wl, cuda_device)
    sets = synth.row_sets(wl, 1)
    lr32 = float(np.float32(wl.lr))
    for t in range(1, steps + 1):
        G = synth.dense_grad(wl, 1, t, cuda_device, scales=scales, sets=sets)
        emb.step_dense(W, G, wl.lr, t)
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, lr32, t)
    torch.cuda.synchronize()
    st = emb.state.cpu().numpy()
    check_state(st[:V], r, "r")
    check_state(st[V:], c, "c")
    d = bf16_ulp_distance(w_to_host(W), Wo)
    report(wl.name, steps=steps, max_ulp=int(d.max()), frac_differ=f"{(d > 0).mean():.3g}",
           frac_over_1ulp=f"{(d > 1).mean():.3g}")
    assert d.max() <= steps
    assert (d > 1).mean() <= 0.01


def test_sparse_trajectory(cuda_device):
    V, D, N, steps = 5000, 128, 3000, 8
    wl = synth.Workload("sparse_small", V, D, "bf16", steps, kind="sparse", N=N)
    emb = Ember(V, D, wdtype="bf16", max_sparse_N=N, device=cuda_device)
    W = synth.init_weights(wl, 2, cuda_device)
    Wo = w_to_host(W)
    r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
    lr32 = float(np.float32(wl.lr))
    for t in range(1, steps + 1):
        ids, rows = synth.sparse_batch(wl, 2, t, cuda_device)
        emb.step_sparse(W, ids, rows, wl.lr, t)
        oracle.step_sparse(Wo, ids.cpu().numpy(), rows.cpu().numpy(), r, c, lr32, t)
    torch.cuda.synchronize()
    assert emb.device_status() == 0
    st = emb.state.cpu().numpy()
    check_state(st[:V], r, "r")
    check_state(st[V:], c, "c")
    d = bf16_ulp_distance(w_to_host(W), Wo)
    report(wl.name, steps=steps, max_ulp=int(d.max()), frac_differ=f"{(d > 0).mean():.3g}",
           frac_over_1ulp=f"{(d > 1).mean():.3g}")
    assert d.max() <= steps
    assert (d > 1).mean() <= 0.01


def test_lmhead_trajectory(cuda_device):
    """The fused LM-head step, ungated against the oracle's step on the same
    G each time (G itself is checked per step by the LM-head tests)."""
    V, D, T, steps = 1000, 328, 100, 6
    emb = Ember(V, D, wdtype="f32", device=cuda_device)
    W = torch.randn(V, D, device=cuda_device, generator=torch.Generator(device=cuda_device).manual_seed(3)) * 0.02
    Wo = w_to_host(W)
    r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
    G = torch.empty(V, D, device=cuda_device)
    lr = 1e-3
    for t in range(1, steps + 1):
        dl, h = synth.lmhead_inputs(V, D, T, 5, t, cuda_device)
        emb.step_lmhead(W, dl, h, G, lr, t)
        torch.cuda.synchronize()
        oracle.step_dense(Wo, G.cpu().numpy(), r, c, float(np.float32(lr)), t)
    st = emb.state.cpu().numpy()
    check_state(st[:V], r, "r")
    check_state(st[V:], c, "c")
    rel = np.abs(w_to_host(W).astype(np.float64) - Wo) / np.maximum(np.abs(Wo), lr)
    report("lmhead 1000x328 T=100", steps=steps, max_rel_W=f"{rel.max():.3g}")
    assert rel.max() <= steps * 1e-5
