"""A table of more than 2^31 elements, at the largest V the ABI accepts.

V = 2^31 - 1 rows of D = 4 columns (8.6e9 elements; G alone is 34 GB, W
17 GB), zero gradient except on a few rows at the start, the middle and the
end.  The oracle cannot step a table that size, but the method fixes what
the step must do on it, from a zero state:

* rows whose gradient is zero keep r = 0 and their weights, bit for bit
  (their g^2 is 0 and so is their update g / (...));
* on the K rows with a gradient the step equals the oracle's step on the
  K x D subtable: r_i depends on row i alone; the column moments are means
  over all V rows, c = (K / V) c_sub, and the means of rhat and chat scale
  the same way, s = (K / V) s_sub, so chat_j / s -- and with it every update --
  is the subtable's (the update is dimensionless: appendix "Outer Product
  Unit Alignment").

Each step is gated: the oracle starts from the GPU's own rows, its r and its
c scaled by V / K.  The test needs about 70 GB of device memory.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01455_gb300.ember import Ember
from parity import check_state, check_weights

pytestmark = pytest.mark.gpu

V, D = 2 ** 31 - 1, 4


def test_step_past_two_to_the_31_elements(cuda_device):
    dev = cuda_device
    rows = torch.tensor([0, 1, V // 2, V // 2 + 1, V - 2, V - 1], dtype=torch.int64, device=dev)
    K = rows.numel()
    w0 = 0.02
    emb = Ember(V, D, wdtype="bf16", device=dev)
    W = torch.full((V, D), w0, dtype=torch.bfloat16, device=dev)
    G = torch.zeros((V, D), dtype=torch.float32, device=dev)
    assert W.numel() > 2 ** 31
    gen = torch.Generator(device=dev).manual_seed(31)
    lr = 1e-3
    for t in (1, 2):
        G[rows] = torch.randn(K, D, generator=gen, device=dev) * 1e-3
        Wsub = W[rows].view(torch.int16).cpu().numpy().view(np.uint16).copy()
        W0sub = Wsub.copy()
        r_sub = emb.r[rows].cpu().numpy().copy()
        c_sub = (emb.c.double() * (V / K)).float().cpu().numpy()
        emb.step_dense(W, G, lr, t)
        torch.cuda.synchronize()
        assert emb.device_status() == 0
        oracle.step_dense(Wsub, G[rows].cpu().numpy(), r_sub, c_sub, float(np.float32(lr)), t)
        check_weights(W[rows].view(torch.int16).cpu().numpy().view(np.uint16), Wsub, lr, "W rows", prev=W0sub)
        check_state(emb.r[rows].cpu().numpy(), r_sub, "r rows")
        check_state((emb.c.double() * (V / K)).float().cpu().numpy(), c_sub, "c (times V / K)")
        # every other row: r stays exactly 0, W bit-identical
        assert int(torch.count_nonzero(emb.r)) == K
        touched = W[rows].clone()
        W[rows] = w0
        assert bool(torch.all(W == w0))
        W[rows] = touched
