"""Helpers shared by the GPU parity tests: host copies, tolerances, the
per-step gate against the CPU oracle.

Tolerances (the stated bar): fp32 state and fp32 weights within a relative
error of 1e-5 (weights relative to max(|W|, lr), the size of one update;
state relative to |ref|, with zeros exact); bf16 weights within 1 ulp.
"""
import numpy as np
import torch

import oracle

REL_TOL = 1e-5
BF16_ULPS = 1


def w_to_host(W):
    """numpy copy of W: float32, or bfloat16 bit patterns as uint16."""
    if W.dtype == torch.bfloat16:
        return W.detach().view(torch.int16).cpu().numpy().view(np.uint16).copy()
    return W.detach().cpu().numpy().copy()


def bf16_ordinal(bits):
    b = bits.astype(np.int64)
    mag = b & 0x7FFF
    return np.where(b & 0x8000, -mag, mag)


def bf16_ulp_distance(a, b):
    return np.abs(bf16_ordinal(a) - bf16_ordinal(b))


def check_weights(got, want, lr, what="W"):
    if got.dtype == np.uint16:
        d = bf16_ulp_distance(got, want)
        worst = int(d.max()) if d.size else 0
        assert worst <= BF16_ULPS, f"{what}: {worst} bf16 ulps apart (at {np.unravel_index(d.argmax(), d.shape)})"
        return {"max_ulp": worst, "frac_differ": float((d > 0).mean()) if d.size else 0.0}
    g = got.astype(np.float64)
    w = want.astype(np.float64)
    rel = np.abs(g - w) / np.maximum(np.abs(w), abs(lr))
    worst = float(rel.max()) if rel.size else 0.0
    assert worst <= REL_TOL, f"{what}: relative error {worst:.3g}"
    return {"max_rel": worst}


def check_state(got, want, what="state"):
    g = got.astype(np.float64)
    w = want.astype(np.float64)
    zero = w == 0
    assert np.all(g[zero] == 0), f"{what}: nonzero where the oracle has exact zeros"
    rel = np.abs(g - w) / np.maximum(np.abs(w), 1e-30)
    worst = float(rel.max()) if rel.size else 0.0
    assert worst <= REL_TOL, f"{what}: relative error {worst:.3g} at {int(rel.argmax())}"
    return {"max_rel": worst}


def oracle_kwargs(opt):
    return dict(beta2=opt.beta2, eps=opt.eps, maximize=opt.maximize,
                bias_correction=opt.bias_correction, variant=opt.variant)


class Opt:
    """Hyper-parameters of one run, in the oracle's and the binding's terms."""

    def __init__(self, beta2=0.999, eps=1e-8, maximize=False, bias_correction=True, variant="full"):
        self.beta2, self.eps, self.maximize = beta2, eps, maximize
        self.bias_correction, self.variant = bias_correction, variant


def gated_dense_step(emb, W, G, lr, t, opt):
    """Run one GPU step and the oracle's step from the same W_{t-1}, state_{t-1}
    and G; compare W_t and the state.  Returns error statistics."""
    V = emb.V
    W0 = w_to_host(W)
    st0 = emb.state.cpu().numpy().copy()
    Gh = G.detach().cpu().numpy()
    emb.step_dense(W, G, lr, t)
    torch.cuda.synchronize()
    r, c = st0[:V].copy(), st0[V:].copy()
    Wo = W0.copy()
    oracle.step_dense(Wo, Gh, r, c, float(np.float32(lr)), t, **oracle_kwargs(opt))
    st = emb.state.cpu().numpy()
    stats = {}
    stats["r"] = check_state(st[:V], r, "r")
    stats["c"] = check_state(st[V:], c, "c")
    stats["W"] = check_weights(w_to_host(W), Wo, lr)
    return stats
