"""Helpers shared by the GPU parity tests: host copies, tolerances, the
per-step gate against the CPU oracle.

Tolerances (the stated bar): fp32 state and fp32 weights within a relative
error of 1e-5 (weights relative to max(|W|, lr, |W_t - W_{t-1}|), the size
of the weight or of one update; state relative to |ref|, with zeros exact);
bf16 weights within 1 ulp.

The size of one update is lr |u| with u = g / (sqrt(vtil) + eps)
(Algorithm 1).  With the bias correction on, |u| is of order 1 and lr
stands for it; without it (the ablation of Section 2.1), vtil at step t is
(1 - beta2^t) times smaller and |u| reaches 1/sqrt(1 - beta2^t), about 32
at t = 1 for beta2 = 0.999.  An fp32 error of a few ulps of that update,
where the new weight nearly cancels to zero, is then far above 1e-5 lr; the
floor therefore also takes the oracle's own step |W_t - W_{t-1}| when the
previous weights are given.

One refinement of the bf16 bar, derived from the arithmetic: the kernel forms
W - lr u in fp32 (the paper fixes no precision), so u carries a relative
error of a few fp32 ulps (~3e-7).  Where the new weight nearly cancels to
zero, a bf16 ulp of the result is smaller than that error (|W_new| below
~4e-7 for |W| ~ 0.02), and no fp32 computation can promise 1 ulp there.
Those elements are held to the fp32-weight bar instead: |got - want| <=
1e-5 max(|want|, lr).  The share of elements that pass only that way is
returned so that the tests can bound it.
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


def check_weights(got, want, lr, what="W", prev=None):
    """`prev`: the weights before the step (same dtype), whose difference from
    `want` is the oracle's own step size."""
    if got.dtype == np.uint16:
        d = bf16_ulp_distance(got, want)
        far = d > BF16_ULPS
        n_far = int(far.sum())
        if n_far:
            assert n_far <= max(2, 1e-3 * d.size), f"{what}: {n_far} elements more than 1 bf16 ulp apart"
            g = oracle.bf16_to_float64(got[far])
            w = oracle.bf16_to_float64(want[far])
            floor = np.maximum(np.abs(w), abs(lr))
            if prev is not None:
                floor = np.maximum(floor, np.abs(w - oracle.bf16_to_float64(prev[far])))
            rel = np.abs(g - w) / floor
            k = int(rel.argmax())
            assert rel[k] <= REL_TOL, (
                f"{what}: {int(d.max())} bf16 ulps apart, {g[k]!r} vs {w[k]!r} "
                f"(relative {rel[k]:.3g} of max(|W|, lr))")
        return {"max_ulp": int(d.max()) if d.size else 0,
                "frac_differ": float((d > 0).mean()) if d.size else 0.0,
                "frac_near_zero_fallback": n_far / max(d.size, 1)}
    g = got.astype(np.float64)
    w = want.astype(np.float64)
    floor = np.maximum(np.abs(w), abs(lr))
    if prev is not None:
        floor = np.maximum(floor, np.abs(w - prev.astype(np.float64)))
    rel = np.abs(g - w) / floor
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
    stats["W"] = check_weights(w_to_host(W), Wo, lr, prev=W0)
    return stats
