"""Seeded synthetic inputs shaped like the paper's token-table workloads.

Input generation only: nothing here computes any part of the Ember step.
The tests and the benchmark draw every input from these functions; the CUDA
library and the CPU oracle then both consume the same arrays.

Recipe (the paper trains GPT-2 / Pythia / Qwen token tables on FineWeb,
Alpaca and Countdown; none of that data is used or needed):

* token id = frequency rank.  Row i of a dense gradient is i.i.d.
  N(0, s_i^2) with s_i = sigma0 (i + 1)^-0.5, sigma0 = 1e-3, so the row
  energy falls with the rank the way the squared-frequency row Fisher of the
  appendix "The Fisher is proportional to inverse frequency squared" does for
  a Zipf token distribution;
* W_0 is i.i.d. N(0, 0.02^2), stored as the table's weight type;
* the tied-table workload has round(0.001 V) rows (a fixed seeded set) whose
  gradient is exactly zero at every step (never-seen tokens);
* the large LM-head workload draws 1 % of its rows (a fixed seeded set) as
  s_i * t_3 with t_3 = Z / sqrt(chi^2_3 / 3) built from four normals
  (heavy-tailed rows);
* the sparse workload draws N token ids per step i.i.d. from Zipf(1.1)
  truncated to [0, V) (p_k proportional to (k + 1)^-1.1, inverse CDF in
  fp64 on uniform draws; duplicates kept) and one gradient row per
  occurrence, i.i.d. N(0, (1e-4)^2);
* the LM-head gradient workload draws, per step, the two factors of the
  head's gradient for T tokens (appendix "Decomposing the Squared
  Gradient"): logits i.i.d. N(0, 2^2) per token, the softmax error
  dlogits[t] = (softmax(logits_t) - onehot(y_t)) / T with targets y_t
  i.i.d. Zipf(1.1) as above, and hidden states i.i.d. N(0, 1); both are
  stored as bfloat16.  G = dlogits^T H then has the Zipf row-energy profile
  of a trained head (frequent targets carry the largest rows).

Seeds: W_0 uses seed * 1_000_003; step t (t >= 1) uses
seed * 1_000_003 + t on a generator of the target device; the fixed row sets
use a CPU generator seeded with `seed`.
"""
from dataclasses import dataclass

import torch

SIGMA0 = 1e-3
W_STD = 0.02
SPARSE_STD = 1e-4
ZIPF_S = 1.1


@dataclass(frozen=True)
class Workload:
    name: str
    V: int
    D: int
    wdtype: str          # "f32" or "bf16"
    steps: int
    kind: str = "dense"  # "dense" or "sparse"
    N: int = 0           # ids per sparse step
    zero_frac: float = 0.0
    heavy_frac: float = 0.0
    lr: float = 1e-3
    T: int = 0           # tokens per LM-head gradient


WORKLOADS = {
    w.name: w for w in [
        Workload("dense_v1024_d64_f32", 1024, 64, "f32", 10),
        Workload("dense_v32000_d4096_bf16", 32000, 4096, "bf16", 100),
        Workload("dense_tied_v151936_d896_bf16", 151936, 896, "bf16", 100, zero_frac=0.001),
        Workload("sparse_v262144_d2048_bf16_n32768", 262144, 2048, "bf16", 100, kind="sparse",
                 N=8 * 4096),
        Workload("dense_lmhead_v128256_d8192_bf16", 128256, 8192, "bf16", 50, heavy_frac=0.01),
        Workload("lmhead_grad_v128256_d8192_t4096_bf16", 128256, 8192, "bf16", 20, kind="lmhead",
                 T=4096),
        # a quarter of the head's rows: the size the detailed profiles use
        Workload("lmhead_grad_v32768_d8192_t4096_bf16", 32768, 8192, "bf16", 20, kind="lmhead", T=4096),
        Workload("dense_v32768_d8192_bf16", 32768, 8192, "bf16", 20, heavy_frac=0.01),
        # an LM head wider than one CTA's row (a 128256-token vocabulary at
        # hidden size 16384): the step runs in two column panels
        Workload("dense_wide_v128256_d16384_bf16", 128256, 16384, "bf16", 20, heavy_frac=0.01),
    ]
}
# The five workloads of the optimizer step, in the order they are listed for
# the paper's method (the others are the LM-head gradient, the wide table and
# the quarter-size tables the detailed profiles use).
ORDER = ["dense_v1024_d64_f32", "dense_v32000_d4096_bf16", "dense_tied_v151936_d896_bf16",
         "sparse_v262144_d2048_bf16_n32768", "dense_lmhead_v128256_d8192_bf16"]
LOGIT_STD = 2.0


def torch_wdtype(wl):
    return torch.bfloat16 if wl.wdtype == "bf16" else torch.float32


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def init_weights(wl, seed=0, device="cuda"):
    """W_0 ~ N(0, 0.02^2), V x D, in the workload's weight type."""
    g = _gen(device, seed * 1_000_003)
    W = torch.randn(wl.V, wl.D, generator=g, device=device, dtype=torch.float32) * W_STD
    return W.to(torch_wdtype(wl))


def row_sets(wl, seed=0):
    """(zero_rows, heavy_rows): fixed seeded row index sets (CPU int64)."""
    g = _gen("cpu", seed)
    perm = torch.randperm(wl.V, generator=g)
    nz = int(round(wl.zero_frac * wl.V))
    nh = int(round(wl.heavy_frac * wl.V))
    return perm[:nz].sort().values, perm[nz:nz + nh].sort().values


def row_scales(wl, device="cuda"):
    """s_i = sigma0 (i + 1)^-0.5 as a V x 1 fp32 column."""
    i = torch.arange(wl.V, device=device, dtype=torch.float64)
    return (SIGMA0 * (i + 1.0) ** -0.5).to(torch.float32).unsqueeze(1)


def dense_grad(wl, seed, t, device="cuda", out=None, scales=None, sets=None):
    """The V x D fp32 gradient of step t (t >= 1)."""
    g = _gen(device, seed * 1_000_003 + t)
    if out is None:
        out = torch.empty(wl.V, wl.D, device=device, dtype=torch.float32)
    torch.randn(out.shape, generator=g, device=device, dtype=torch.float32, out=out)
    out.mul_(scales if scales is not None else row_scales(wl, device))
    zero_rows, heavy_rows = sets if sets is not None else row_sets(wl, seed)
    if len(heavy_rows):
        hr = heavy_rows.to(device)
        z = torch.randn(len(hr), wl.D, generator=g, device=device, dtype=torch.float32)
        chi = torch.randn(3, len(hr), wl.D, generator=g, device=device, dtype=torch.float32)
        t3 = z / torch.sqrt((chi * chi).sum(0) / 3.0)
        out[hr] = t3 * (scales if scales is not None else row_scales(wl, device))[hr]
    if len(zero_rows):
        out[zero_rows.to(device)] = 0.0
    return out


_ZIPF_CDF = {}


def zipf_cdf(V, device):
    key = (V, str(device))
    if key not in _ZIPF_CDF:
        p = (torch.arange(V, device=device, dtype=torch.float64) + 1.0) ** -ZIPF_S
        cdf = torch.cumsum(p, 0)
        cdf /= cdf[-1].clone()
        cdf[-1] = 1.0
        _ZIPF_CDF[key] = cdf
    return _ZIPF_CDF[key]


def sparse_batch(wl, seed, t, device="cuda", N=None):
    """(ids int64 [N], rows fp32 [N, D]) of sparse step t (t >= 1)."""
    N = wl.N if N is None else N
    g = _gen(device, seed * 1_000_003 + t)
    u = torch.rand(N, generator=g, device=device, dtype=torch.float64)
    ids = torch.searchsorted(zipf_cdf(wl.V, device), u, right=True).clamp_(max=wl.V - 1)
    rows = torch.randn(N, wl.D, generator=g, device=device, dtype=torch.float32) * SPARSE_STD
    return ids.to(torch.int64), rows


def lmhead_inputs(V, D, T, seed, t, device="cuda", chunk=512):
    """(dlogits bf16 [T, V], hidden bf16 [T, D]) of step t (t >= 1): the
    softmax error of T tokens, already divided by T, and their hidden states."""
    g = _gen(device, seed * 1_000_003 + t)
    u = torch.rand(T, generator=g, device=device, dtype=torch.float64)
    y = torch.searchsorted(zipf_cdf(V, device), u, right=True).clamp_(max=V - 1)
    dl = torch.empty(T, V, device=device, dtype=torch.bfloat16)
    for t0 in range(0, T, chunk):
        t1 = min(T, t0 + chunk)
        z = torch.randn(t1 - t0, V, generator=g, device=device, dtype=torch.float32) * LOGIT_STD
        q = torch.softmax(z, dim=1)
        q[torch.arange(t1 - t0, device=device), y[t0:t1]] -= 1.0
        dl[t0:t1] = (q / T).to(torch.bfloat16)
    hidden = torch.randn(T, D, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    return dl, hidden
