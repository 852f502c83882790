"""Out-of-bounds writes: W, G, the rows and the state sit between canary
regions, and every step must leave the canaries bit-identical.  Shapes are
ragged (D not a multiple of 4, V not a multiple of the CTA count) so that
every tail path runs."""
import pytest
import torch

from paper_2607_01455_gb300.ember import Ember

pytestmark = pytest.mark.gpu

GUARD = 4096  # elements of canary on each side


def guarded(n, dtype, device, fill):
    """A tensor of n elements with GUARD canary elements on both sides."""
    buf = torch.empty(n + 2 * GUARD, dtype=dtype, device=device)
    buf.fill_(fill)
    return buf, buf[GUARD:GUARD + n]


def canaries_intact(buf, n, fill):
    return bool(torch.all(buf[:GUARD] == fill)) and bool(torch.all(buf[GUARD + n:] == fill))


@pytest.mark.parametrize("V,D,wdtype,variant", [
    (305, 33, "bf16", "full"), (1000, 127, "f32", "full"), (7, 1, "bf16", "full"),
    (777, 1028, "bf16", "full"), (40, 8192, "bf16", "full"), (513, 203, "bf16", "row"),
    (300, 8192, "bf16", "row"),
])
def test_dense_steps_stay_in_bounds(cuda_device, V, D, wdtype, variant):
    wt = torch.bfloat16 if wdtype == "bf16" else torch.float32
    emb = Ember(V, D, wdtype=wdtype, variant=variant, device=cuda_device)
    wbuf, W = guarded(V * D, wt, cuda_device, -7.0)
    gbuf, G = guarded(V * D, torch.float32, cuda_device, 9.0)
    W.copy_(torch.randn(V * D, device=cuda_device).to(wt) * 0.02)
    for t in (1, 2):
        G.copy_(torch.randn(V * D, device=cuda_device) * 1e-3)
        emb.step_dense(W.view(V, D), G.view(V, D), 1e-3, t)
    torch.cuda.synchronize()
    assert canaries_intact(wbuf, V * D, -7.0)
    assert canaries_intact(gbuf, V * D, 9.0)
    assert emb.device_status() == 0


@pytest.mark.parametrize("V,D,N", [(1000, 33, 3001), (5000, 127, 1025), (300, 2048, 4097)])
def test_sparse_steps_stay_in_bounds(cuda_device, V, D, N):
    emb = Ember(V, D, wdtype="bf16", max_sparse_N=N, device=cuda_device)
    wbuf, W = guarded(V * D, torch.bfloat16, cuda_device, -7.0)
    rbuf, rows = guarded(N * D, torch.float32, cuda_device, 9.0)
    W.copy_(torch.randn(V * D, device=cuda_device).to(torch.bfloat16) * 0.02)
    for t in (1, 2):
        ids = (torch.rand(N, device=cuda_device) ** 2 * V).long()
        rows.copy_(torch.randn(N * D, device=cuda_device) * 1e-4)
        emb.step_sparse(W.view(V, D), ids, rows.view(N, D), 1e-3, t)
    torch.cuda.synchronize()
    assert canaries_intact(wbuf, V * D, -7.0)
    assert canaries_intact(rbuf, N * D, 9.0)
    assert emb.device_status() == 0


def test_from_host_step_stays_in_bounds(cuda_device):
    V, D = 301, 96
    emb = Ember(V, D, wdtype="bf16", device=cuda_device)
    wbuf, W = guarded(V * D, torch.bfloat16, cuda_device, -7.0)
    sbuf, stage = guarded(V * D, torch.float32, cuda_device, 5.0)
    W.copy_(torch.randn(V * D, device=cuda_device).to(torch.bfloat16) * 0.02)
    Gh = (torch.randn(V, D) * 1e-3).pin_memory()
    emb.step_dense_from_host(W.view(V, D), Gh, stage.view(V, D), 1e-3, 1)
    torch.cuda.synchronize()
    assert canaries_intact(wbuf, V * D, -7.0)
    assert canaries_intact(sbuf, V * D, 5.0)
