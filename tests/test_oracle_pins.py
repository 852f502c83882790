"""Pins for the CPU oracle: facts fixed by the paper or by mathematics, not by
the oracle's own formula.

Each test names the passage of "Token Geometry" (arXiv 2607.01455) it rests on
and the mistakes it is there to catch.  All run on the CPU (-m "not gpu").
"""
import bisect
import collections
import json
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def f32_ulp(x):
    return np.spacing(np.abs(np.asarray(x, np.float32))).astype(np.float64)


def exact_rank1_factors(rng, n, lo=-6, hi=3):
    """Values (+-1, 3, 5 or 7) * 2^k: products of two of them are exact in fp32."""
    mant = rng.choice([1.0, 3.0, 5.0, 7.0], size=n)
    sign = rng.choice([-1.0, 1.0], size=n)
    expo = rng.integers(lo, hi, size=n)
    return sign * mant * np.exp2(expo)


# --------------------------------------------------------------------------
# bfloat16 rounding (the storage type of W).  Round to nearest, ties to even.
# --------------------------------------------------------------------------

def _all_finite_bf16():
    bits = np.arange(0, 0x7F80, dtype=np.uint32).astype(np.uint16)  # +0 .. max finite
    vals = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return bits, vals


def _brute_round_bf16(x, bits, vals):
    """Nearest representable bfloat16 by search over all of them; ties to the
    even bit pattern; past (max + half its spacing) to infinity."""
    a = abs(x)
    top = vals[-1] + (vals[-1] - vals[-2]) / 2
    if a >= top:
        b = 0x7F80
    else:
        k = bisect.bisect_left(vals, a)
        if k < len(vals) and vals[k] == a:
            b = int(bits[k])
        else:
            lo, hi = k - 1, k
            dl, dh = a - vals[lo], vals[hi] - a
            if dl < dh:
                b = int(bits[lo])
            elif dh < dl:
                b = int(bits[hi])
            else:
                b = int(bits[lo]) if int(bits[lo]) % 2 == 0 else int(bits[hi])
    return b | (0x8000 if np.signbit(x) else 0)


def test_bf16_rounding_matches_brute_force_search():
    rng = np.random.default_rng(1)
    bits, vals = _all_finite_bf16()
    xs = list(rng.standard_normal(3000) * np.exp2(rng.integers(-140, 128, 3000)))
    xs += [vals[k] + (vals[k + 1] - vals[k]) / 2 for k in rng.integers(0, len(vals) - 1, 300)]
    xs += [-(vals[k] + (vals[k + 1] - vals[k]) / 2) for k in rng.integers(0, len(vals) - 1, 300)]
    xs += [0.0, -0.0, 1e-45, 2.0 ** -133, 2.0 ** -134, 3 * 2.0 ** -135, 3.4e38, 3.3895e38, 1e39]
    xs = np.array(xs, np.float64)
    got = oracle.round_bf16(xs)
    want = np.array([_brute_round_bf16(x, bits, vals) for x in xs], np.uint16)
    np.testing.assert_array_equal(got, want)


def test_bf16_rounding_matches_torch_on_fp32_values():
    rng = np.random.default_rng(2)
    x32 = (rng.standard_normal(200000) * np.exp2(rng.integers(-130, 127, 200000))).astype(np.float32)
    want = torch.from_numpy(x32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.round_bf16(x32.astype(np.float64)), want)
    np.testing.assert_array_equal(oracle.bf16_to_float64(want),
                                  torch.from_numpy(want.view(np.int16)).view(torch.bfloat16)
                                  .to(torch.float64).numpy())


# --------------------------------------------------------------------------
# Reduction to a textbook optimizer.  With D = 1 the column factor is the
# grand mean, mean(rhat) equals it (appendix "Outer Product Unit Alignment"),
# so s = chat and vtil_i = rhat_i: Ember is Adam with the first moment
# replaced by the instantaneous gradient (Section 2.1, "completely removing
# the first moment's EMA"), i.e. torch.optim.Adam with beta1 = 0.  The same
# holds for V = 1 by the row/column symmetry of Algorithm 1.
# Catches: EMA weights swapped, wrong bias-correction power, eps inside the
# square root, a missing square root, a wrong sign, the wrong axis.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("shape", [(9, 1), (1, 7)])
@pytest.mark.parametrize("variant", ["full", "row", "col"])
def test_single_row_or_column_is_adam_without_first_moment(shape, variant):
    if (variant, shape) in {("row", (1, 7)), ("col", (9, 1))}:
        pytest.skip("that variant pools the whole vector; not elementwise Adam")
    rng = np.random.default_rng(3)
    beta2, eps, lr, steps = 0.9, 1e-3, 1e-2, 7
    W0 = rng.standard_normal(shape).astype(np.float32)
    grads = [(rng.standard_normal(shape) * np.exp2(rng.integers(-8, 3, shape))).astype(np.float32)
             for _ in range(steps)]

    p = torch.nn.Parameter(torch.from_numpy(W0.astype(np.float64)))
    opt = torch.optim.Adam([p], lr=lr, betas=(0.0, beta2), eps=eps)
    W = W0.copy()
    r = np.zeros(shape[0], np.float32)
    c = np.zeros(shape[1], np.float32)
    for t, g in enumerate(grads, start=1):
        p.grad = torch.from_numpy(g.astype(np.float64))
        opt.step()
        oracle.step_dense(W, g, r, c, lr, t, beta2=beta2, eps=eps, variant=variant)
        ref = p.detach().numpy()
        # fp32 storage of W and of the state; a formula slip moves W by ~lr.
        np.testing.assert_allclose(W, ref, rtol=0, atol=t * (4 * f32_ulp(ref).max() + 1e-7 * lr))


# --------------------------------------------------------------------------
# Exactness of the geometric-mean normaliser (appendix "Outer Product Unit
# Alignment", paragraph "Exactness"): if g_ij^2 = a_i^2 b_j^2 then
# vtil_ij = a_i^2 b_j^2, so the first step is alpha * g / (|g| + eps) -- a
# z-score cast to one bit, i.e. signSGD (Section 2.2, "Interpreting the
# metric").  A gradient repeated every step keeps rhat fixed, so every step
# moves by the same amount.
# Catches: missing or doubled bias correction, sum instead of mean over a
# row, no normaliser, s without its square root, eps misplaced, sign errors.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("beta2", [0.999, 0.9])
def test_rank_one_gradient_gives_sign_update(beta2):
    rng = np.random.default_rng(4)
    V, D, lr, eps, steps = 7, 5, 1e-3, 1e-8, 5
    a = exact_rank1_factors(rng, V)
    b = exact_rank1_factors(rng, D)
    a[2] = 2.0 ** -27          # |g| near eps in that row: eps must sit outside the sqrt
    G = np.outer(a, b).astype(np.float32)
    assert np.array_equal(G.astype(np.float64), np.outer(a, b))  # exactly rank one
    W = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    r = np.zeros(V, np.float32)
    c = np.zeros(D, np.float32)
    g = G.astype(np.float64)
    want_u = g / (np.abs(g) + eps)
    for t in range(1, steps + 1):
        W_prev = W.copy()
        oracle.step_dense(W, G, r, c, lr, t, beta2=beta2, eps=eps)
        want = (W_prev.astype(np.float64) - lr * want_u).astype(np.float32)
        np.testing.assert_allclose(W, want, rtol=0, atol=f32_ulp(want).max() + 1e-6 * lr)
    # and the state is the closed form too: r_t = (1 - beta2^t) a_i^2 mean(b^2)
    bc = 1 - beta2 ** steps
    np.testing.assert_allclose(r, bc * a ** 2 * np.mean(b ** 2), rtol=1e-6 * steps)
    np.testing.assert_allclose(c, bc * b ** 2 * np.mean(a ** 2), rtol=1e-6 * steps)


def test_two_step_ema_closed_form():
    """G_1 = a b^T then G_2 = kappa a b^T.  Algorithm 1 gives
    rhat_2 = (beta2 + kappa^2)/(1 + beta2) * a_i^2 mean(b^2) and the same
    factor k on chat and on s, so sqrt(vtil) = sqrt(k) |a_i b_j| and the
    second update is alpha kappa g / (sqrt(k) |g| + eps).
    Catches: beta2 and 1-beta2 swapped, bias correction with t-1 or t+1,
    the current gradient left out of the second moment."""
    rng = np.random.default_rng(5)
    V, D, lr, eps, beta2, kappa = 6, 11, 1e-2, 1e-8, 0.9, 3.0
    a = exact_rank1_factors(rng, V)
    b = exact_rank1_factors(rng, D)
    G1 = np.outer(a, b).astype(np.float32)
    W = np.zeros((V, D), np.float32)
    r = np.zeros(V, np.float32)
    c = np.zeros(D, np.float32)
    oracle.step_dense(W, G1, r, c, lr, 1, beta2=beta2, eps=eps)
    W1 = W.copy()
    oracle.step_dense(W, (kappa * G1).astype(np.float32), r, c, lr, 2, beta2=beta2, eps=eps)
    k = (beta2 + kappa ** 2) / (1 + beta2)
    g = G1.astype(np.float64)
    want = (W1.astype(np.float64) - lr * kappa * g / (np.sqrt(k) * np.abs(g) + eps)).astype(np.float32)
    np.testing.assert_allclose(W, want, rtol=0, atol=2 * f32_ulp(want).max() + 1e-6 * lr)


# --------------------------------------------------------------------------
# mean(rhat) == mean(chat) identically: both are the grand mean of g^2
# (appendix "Outer Product Unit Alignment").
# Catches: dividing the row sums by V and the column sums by D.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("bias_correction", [True, False])
def test_row_and_column_means_agree(bias_correction):
    rng = np.random.default_rng(6)
    V, D = 13, 6
    W = np.zeros((V, D), np.float32)
    r = np.zeros(V, np.float32)
    c = np.zeros(D, np.float32)
    for t in range(1, 6):
        G = (rng.standard_normal((V, D)) * np.exp2(rng.integers(-10, 2, (V, 1)))).astype(np.float32)
        d = oracle.step_dense(W, G, r, c, 1e-3, t, beta2=0.95, bias_correction=bias_correction)
        assert abs(d["rbar"] - d["cbar"]) <= 1e-6 * d["rbar"]
        assert d["s"] == pytest.approx(d["rbar"], rel=1e-6)


# --------------------------------------------------------------------------
# The update is dimensionless (Section 2.2, "Interpreting the metric";
# appendix "Outer Product Unit Alignment"): with eps = 0, scaling every
# gradient by 2^m leaves the weights bit-identical, since powers of two pass
# exactly through squares, means, the fp32 state, sqrt and division.
# Catches: wrong power of s or of the row/column factors.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("wdtype", [np.float32, np.uint16])
@pytest.mark.parametrize("m", [7, -9])
def test_power_of_two_gradient_scale_invariance(wdtype, m):
    rng = np.random.default_rng(7)
    V, D = 10, 12
    W0 = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    if wdtype == np.uint16:
        W0 = oracle.round_bf16(W0.astype(np.float64))
    Wa, Wb = W0.copy(), W0.copy()
    ra, ca = np.zeros(V, np.float32), np.zeros(D, np.float32)
    rb, cb = ra.copy(), ca.copy()
    for t in range(1, 5):
        G = (rng.standard_normal((V, D)) * 1e-3).astype(np.float32)
        oracle.step_dense(Wa, G, ra, ca, 1e-3, t, eps=0.0)
        oracle.step_dense(Wb, (G * np.float32(2.0 ** m)), rb, cb, 1e-3, t, eps=0.0)
        np.testing.assert_array_equal(Wa, Wb)
        np.testing.assert_array_equal(ra * np.float32(2.0 ** (2 * m)), rb)


# --------------------------------------------------------------------------
# Sign: Algorithm 1 ascends; the library descends.  Because the denominator
# sees g only through g^2, ascending on -G equals descending on G exactly.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("wdtype", [np.float32, np.uint16])
def test_maximize_on_negated_gradient_equals_descent(wdtype):
    rng = np.random.default_rng(8)
    V, D = 8, 9
    W0 = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    if wdtype == np.uint16:
        W0 = oracle.round_bf16(W0.astype(np.float64))
    Wa, Wb = W0.copy(), W0.copy()
    ra, ca = np.zeros(V, np.float32), np.zeros(D, np.float32)
    rb, cb = ra.copy(), ca.copy()
    for t in range(1, 4):
        G = (rng.standard_normal((V, D)) * 1e-3).astype(np.float32)
        oracle.step_dense(Wa, G, ra, ca, 1e-3, t)
        oracle.step_dense(Wb, -G, rb, cb, 1e-3, t, maximize=True)
        np.testing.assert_array_equal(Wa, Wb)
        np.testing.assert_array_equal(ra, rb)
        np.testing.assert_array_equal(ca, cb)


def test_descent_moves_against_the_gradient():
    rng = np.random.default_rng(9)
    V, D = 5, 4
    G = (rng.standard_normal((V, D)) * 1e-3).astype(np.float32)
    W = np.zeros((V, D), np.float32)
    oracle.step_dense(W, G, np.zeros(V, np.float32), np.zeros(D, np.float32), 1e-3, 1)
    assert np.all(np.sign(W) == -np.sign(G))
    Wn = np.zeros((V, D), np.float32)
    oracle.step_dense(Wn, -G, np.zeros(V, np.float32), np.zeros(D, np.float32), 1e-3, 1)
    np.testing.assert_array_equal(Wn, -W)


# --------------------------------------------------------------------------
# Row/column symmetry of Algorithm 1: the column rule is the row rule after
# a transpose (Section 2.1: "otherwise identical ... following a transpose").
# Catches: a transposed operand or index anywhere in the step.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("variant,tvariant", [("full", "full"), ("row", "col"), ("col", "row")])
def test_transpose_duality(variant, tvariant):
    rng = np.random.default_rng(10)
    V, D = 9, 4
    W = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    Wt = np.ascontiguousarray(W.T)
    r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
    rt, ct = np.zeros(D, np.float32), np.zeros(V, np.float32)
    for t in range(1, 4):
        G = (rng.standard_normal((V, D)) * np.exp2(rng.integers(-6, 2, (V, 1)))).astype(np.float32)
        oracle.step_dense(W, G, r, c, 1e-2, t, variant=variant)
        oracle.step_dense(Wt, np.ascontiguousarray(G.T), rt, ct, 1e-2, t, variant=tvariant)
        np.testing.assert_allclose(Wt.T, W, rtol=0, atol=2 * f32_ulp(W).max())
        np.testing.assert_allclose(rt, c, rtol=1e-6)
        np.testing.assert_allclose(ct, r, rtol=1e-6)


# --------------------------------------------------------------------------
# Rows that never receive gradient (never-seen tokens of a tied table):
# r_i stays exactly 0 and the weights of that row never move, since
# u = 0 / (0 + eps) = 0 (Algorithm 1's update).
# A step with G = 0 after others decays both moments by beta2 and leaves W.
# --------------------------------------------------------------------------

def test_zero_rows_keep_zero_state_and_weights():
    rng = np.random.default_rng(11)
    V, D = 12, 7
    zero = np.array([0, 5, 11])
    W0 = oracle.round_bf16(rng.standard_normal((V, D)) * 0.02)
    W = W0.copy()
    r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
    for t in range(1, 6):
        G = (rng.standard_normal((V, D)) * 1e-3).astype(np.float32)
        G[zero] = 0.0
        d = oracle.step_dense(W, G, r, c, 1e-3, t)
        assert d["zero_rows"] == len(zero)
    assert np.all(r[zero] == 0.0)
    np.testing.assert_array_equal(W[zero], W0[zero])
    others = np.setdiff1d(np.arange(V), zero)
    assert np.all(W[others] != W0[others])


@pytest.mark.parametrize("wdtype", [np.float32, np.uint16])
def test_zero_gradient_step_only_decays_state(wdtype):
    rng = np.random.default_rng(12)
    V, D, beta2 = 6, 5, 0.999
    W = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    if wdtype == np.uint16:
        W = oracle.round_bf16(W.astype(np.float64))
    r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
    for t in range(1, 4):
        oracle.step_dense(W, (rng.standard_normal((V, D)) * 1e-3).astype(np.float32), r, c, 1e-3, t)
    W3, r3, c3 = W.copy(), r.copy(), c.copy()
    oracle.step_dense(W, np.zeros((V, D), np.float32), r, c, 1e-3, 4, beta2=beta2)
    np.testing.assert_array_equal(W, W3)
    np.testing.assert_array_equal(r, (beta2 * r3.astype(np.float64)).astype(np.float32))
    np.testing.assert_array_equal(c, (beta2 * c3.astype(np.float64)).astype(np.float32))


def test_all_zero_gradient_from_zero_state_is_a_no_op():
    """s = 0 at the first step (nothing seen yet): the update is zero, not NaN."""
    W = np.full((4, 3), 0.5, np.float32)
    r, c = np.zeros(4, np.float32), np.zeros(3, np.float32)
    d = oracle.step_dense(W, np.zeros((4, 3), np.float32), r, c, 1e-3, 1)
    assert d["s"] == 0.0
    assert np.all(W == 0.5) and np.all(r == 0) and np.all(c == 0)


# --------------------------------------------------------------------------
# Ablation variants (Section 2.1 table, appendix "Ablations").
# Row-only at t = 1 divides each row by its RMS (a z-score per token,
# Section 2.1); col-only does the same per column; without bias correction
# the first step of a single parameter is g / (sqrt(1-beta2) |g| + eps).
# --------------------------------------------------------------------------

@pytest.mark.parametrize("variant,axis", [("row", 1), ("col", 0)])
def test_row_and_col_only_first_step_normalises_rms(variant, axis):
    rng = np.random.default_rng(13)
    V, D, lr = 10, 16, 1.0
    G = (rng.standard_normal((V, D)) * np.exp2(rng.integers(-12, 0, (V, 1)))
         * np.exp2(rng.integers(-4, 4, (1, D)))).astype(np.float32)
    W = np.zeros((V, D), np.float32)
    oracle.step_dense(W, G, np.zeros(V, np.float32), np.zeros(D, np.float32), lr, 1,
                      eps=0.0, variant=variant)
    rms = np.sqrt(np.mean(W.astype(np.float64) ** 2, axis=axis))
    np.testing.assert_allclose(rms, 1.0, rtol=1e-6)


def test_no_bias_correction_first_step():
    rng = np.random.default_rng(14)
    beta2, eps = 0.99, 1e-8
    g = (rng.standard_normal((5, 1)) * 1e-2).astype(np.float32)
    W = np.zeros((5, 1), np.float32)
    oracle.step_dense(W, g, np.zeros(5, np.float32), np.zeros(1, np.float32), 1.0, 1,
                      beta2=beta2, eps=eps, bias_correction=False)
    gd = g.astype(np.float64)
    np.testing.assert_allclose(W, -gd / (np.sqrt(1 - beta2) * np.abs(gd) + eps), rtol=1e-6)


# --------------------------------------------------------------------------
# Sparse step (Section 2.2 and appendix "The Fisher is proportional to
# inverse frequency squared"): the embedding gradient is zero except on the
# batch's token rows, and a token seen k times receives the sum of its k
# per-occurrence rows.  Rows with exactly representable sums make the sparse
# oracle and the dense oracle on the scatter-summed gradient agree bit for
# bit; untouched rows keep their weights bit for bit.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("wdtype", [np.float32, np.uint16])
def test_sparse_equals_dense_on_scatter_summed_gradient(wdtype):
    rng = np.random.default_rng(15)
    V, D, N = 40, 6, 64
    W0 = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    if wdtype == np.uint16:
        W0 = oracle.round_bf16(W0.astype(np.float64))
    Ws, Wd = W0.copy(), W0.copy()
    rs, cs = np.zeros(V, np.float32), np.zeros(D, np.float32)
    rd, cd = rs.copy(), cs.copy()
    touched_any = np.zeros(V, bool)
    for t in range(1, 5):
        ids = np.minimum(rng.zipf(1.3, N) - 1, V + 3)   # duplicates and a few ids >= V
        ids[:2] = [-1, V]
        rows = (rng.integers(-64, 65, (N, D)) * 2.0 ** -14).astype(np.float32)
        G = np.zeros((V, D), np.float64)
        ok = (ids >= 0) & (ids < V)
        np.add.at(G, ids[ok], rows[ok].astype(np.float64))
        touched_any[ids[ok]] = True
        oracle.step_sparse(Ws, ids, rows, rs, cs, 1e-3, t)
        oracle.step_dense(Wd, G.astype(np.float32), rd, cd, 1e-3, t)
        np.testing.assert_array_equal(Ws, Wd)
        np.testing.assert_array_equal(rs, rd)
        np.testing.assert_array_equal(cs, cd)
    np.testing.assert_array_equal(Ws[~touched_any], W0[~touched_any])


def test_dedup_matches_counter():
    rng = np.random.default_rng(16)
    V = 1000
    ids = np.concatenate([rng.zipf(1.1, 5000) - 1, [-3, V, V + 7, 0, 0]])
    uniq, counts = oracle.dedup(ids, V)
    want = collections.Counter(int(i) for i in ids if 0 <= i < V)
    assert list(uniq) == sorted(want)
    assert list(counts) == [want[k] for k in sorted(want)]
    u0, c0 = oracle.dedup(np.zeros(0, np.int64), V)
    assert len(u0) == 0 and len(c0) == 0


# --------------------------------------------------------------------------
# State size: Ember keeps exactly V + D fp32 values per token table.  The
# paper's printed sizes follow from (V + D) * 4 bytes per table, against
# AdamW's 2 V D * 4 bytes (Section 3.1 table; Sections 4 and 5.1).
# --------------------------------------------------------------------------

def _in_unit(nbytes, unit):
    return nbytes / {"KiB": 1024, "MiB": 1024 ** 2, "MB": 1e6, "GB": 1e9}[unit]


def test_paper_state_sizes_follow_from_v_plus_d():
    with open(os.path.join(GOLDEN, "state_sizes.json")) as f:
        entries = json.load(f)["entries"]
    for e in entries:
        V, D, n = e["V"], e["D"], e["tables"]
        r, c = np.zeros(V, np.float32), np.zeros(D, np.float32)
        ember_bytes = n * (r.nbytes + c.nbytes)
        adamw_bytes = n * 2 * V * D * 4
        val, unit = e["ember"][0], e["ember"][1]
        tol = 0.05 if "approx" in e["ember"] else 0.005
        assert _in_unit(ember_bytes, unit) == pytest.approx(val, rel=tol), e["model"]
        aval, aunit = e["adamw"]
        assert _in_unit(adamw_bytes, aunit) == pytest.approx(aval, rel=0.01), e["model"]
        if "ratio" in e:
            assert adamw_bytes / ember_bytes == pytest.approx(e["ratio"][0], rel=0.02), e["model"]


# --------------------------------------------------------------------------
# LM-head gradient, the producer of G for an output head (appendix
# "Decomposing the Squared Gradient": per token the outer product of the
# softmax error and the hidden state, summed over the batch).
# --------------------------------------------------------------------------

def _bf16_bits(rng, shape, lo=-8, hi=2):
    """Random finite bfloat16 bit patterns with exponents in [lo, hi)."""
    mant = rng.integers(0, 128, size=shape).astype(np.uint32)
    expo = (rng.integers(lo, hi, size=shape) + 127).astype(np.uint32)
    sign = rng.integers(0, 2, size=shape).astype(np.uint32)
    return ((sign << 15) | (expo << 7) | mant).astype(np.uint16)


def test_lmhead_grad_matches_exact_rational_sum():
    """Brute force in exact rationals: G[v][d] = sum_t delta[t][v] h[t][d].  The
    fp64 result may differ from the exact sum only by the rounding of T - 1
    additions of exactly representable products (bf16 x bf16 fits in 16 bits)."""
    from fractions import Fraction
    rng = np.random.default_rng(11)
    T, V, D = 6, 5, 7
    dl = _bf16_bits(rng, (T, V))
    hd = _bf16_bits(rng, (T, D))
    G, A = oracle.lmhead_grad(dl, hd)
    dv = oracle.bf16_to_float64(dl)
    hv = oracle.bf16_to_float64(hd)
    for v in range(V):
        for d in range(D):
            exact = sum(Fraction(dv[t, v]) * Fraction(hv[t, d]) for t in range(T))
            absum = sum(abs(Fraction(dv[t, v]) * Fraction(hv[t, d])) for t in range(T))
            assert abs(Fraction(G[v, d]) - exact) <= Fraction(T) * Fraction(2) ** -53 * absum
            assert A[v, d] == pytest.approx(float(absum), rel=1e-15)


def test_lmhead_grad_one_hot_errors_gather_hidden_rows():
    """With delta_t = -e_{y_t} (a softmax error whose model probabilities are
    all zero), row v of G is minus the sum of the hidden states of the tokens
    whose target is v; rows of tokens never targeted are exactly zero."""
    rng = np.random.default_rng(12)
    T, V, D = 40, 9, 16
    y = rng.integers(0, V - 2, size=T)  # the last two rows are never targeted
    dl = np.zeros((T, V), np.uint16)
    dl[np.arange(T), y] = 0xBF80  # bfloat16 -1.0
    hd = _bf16_bits(rng, (T, D), lo=-4, hi=1)
    G, _ = oracle.lmhead_grad(dl, hd)
    want = np.zeros((V, D))
    np.add.at(want, y, -oracle.bf16_to_float64(hd))
    np.testing.assert_array_equal(G, want)
    assert not G[V - 2:].any()


def test_lmhead_grad_single_token_is_outer_product():
    rng = np.random.default_rng(13)
    dl = _bf16_bits(rng, (1, 11))
    hd = _bf16_bits(rng, (1, 6))
    G, A = oracle.lmhead_grad(dl, hd)
    outer = np.outer(oracle.bf16_to_float64(dl[0]), oracle.bf16_to_float64(hd[0]))
    np.testing.assert_array_equal(G, outer)
    np.testing.assert_array_equal(A, np.abs(outer))


def test_lmhead_grad_roles_of_the_factors_and_row_selection():
    """Swapping the two factors transposes G (each element is the same sum in
    the same token order); a selected row equals that row of the full G."""
    rng = np.random.default_rng(14)
    T, V, D = 13, 10, 7
    dl = _bf16_bits(rng, (T, V))
    hd = _bf16_bits(rng, (T, D))
    G, _ = oracle.lmhead_grad(dl, hd)
    Gt, _ = oracle.lmhead_grad(hd, dl)
    np.testing.assert_array_equal(Gt, G.T)
    rows = np.array([9, 0, 4])
    Gs, _ = oracle.lmhead_grad(dl, hd, rows=rows)
    np.testing.assert_array_equal(Gs, G[rows])
    # matmul of the exact factors in fp64 agrees to rounding
    ref = oracle.bf16_to_float64(dl).T @ oracle.bf16_to_float64(hd)
    np.testing.assert_allclose(G, ref, rtol=0, atol=1e-12 * np.abs(ref).max())


def test_all_cores_build_gives_the_same_bits():
    """The CPU baseline's OpenMP build of the oracle splits only independent
    loops (rows; blocks of columns, each column still summed over the rows in
    index order), so it must reproduce the plain build bit for bit."""
    rng = np.random.default_rng(11)
    V, D = 517, 203
    W0 = (rng.standard_normal((V, D)) * 0.02).astype(np.float32)
    Gs = [(rng.standard_normal((V, D)) * 1e-3).astype(np.float32) for _ in range(3)]
    assert oracle.threads(4) >= 1
    outs = []
    for all_cores in (False, True):
        Wf, Wh = W0.copy(), oracle.round_bf16(W0.astype(np.float64))
        r1, c1 = np.zeros(V, np.float32), np.zeros(D, np.float32)
        r2, c2 = np.zeros(V, np.float32), np.zeros(D, np.float32)
        for t, G in enumerate(Gs, start=1):
            oracle.step_dense(Wf, G, r1, c1, 1e-3, t, all_cores=all_cores)
            oracle.step_dense(Wh, G, r2, c2, 1e-3, t, variant="col", all_cores=all_cores)
        outs.append((Wf, Wh, r1, c1, r2, c2))
    for a, b in zip(*outs):
        assert np.array_equal(a, b)
