"""The allocation-free dense step against the ordinary one.

ember_step_dense_noalloc serves callers that cannot give the library device
memory (a host allocator with no hook for plugins, a fully reserved memory
budget, a hot path where cudaMalloc would synchronise the device).  It runs
the same kernels as ember_step_dense on the same inputs, only with its
scratch in the library's static array instead of a bound workspace, so W and
the state must come out bit for bit the same, on two calls in a row (the
second call finds the first one's leftovers in the shared array).  This file
is named to be collected last, so a run that stops at its first failure has
run every other test before this one.
"""
import pytest
import torch

from paper_2607_01455_gb300 import ember as E
from parity import check_state, check_weights, w_to_host

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("V,D,wdtype", [(3001, 1024, "bf16"), (777, 8192, "bf16"), (513, 203, "f32")])
def test_noalloc_step_matches_workspace_step(cuda_device, V, D, wdtype):
    ref = E.Ember(V, D, wdtype=wdtype, device=cuda_device)
    h = E.ember_create(V, D, E.ember_hparams_default(), ref.wdtype)
    try:
        state = torch.zeros(E.ember_state_numel(h), dtype=torch.float32, device=cuda_device)
        g = torch.Generator(device=cuda_device)
        g.manual_seed(V + D)
        W0 = torch.randn(V, D, generator=g, device=cuda_device) * 0.02
        W0 = W0.to(torch.bfloat16 if wdtype == "bf16" else torch.float32)
        W_ref, W_na = W0.clone(), W0.clone()
        for t in (1, 2):  # two calls in a row share the library's scratch
            G = torch.randn(V, D, generator=g, device=cuda_device) * 1e-3
            ref.step_dense(W_ref, G, 1e-3, t)
            E.ember_step_dense_noalloc(h, W_na, G, state, 1e-3, t)
            torch.cuda.synchronize()
            # the same kernels on the same inputs: the same bits
            assert torch.equal(W_na.view(torch.int16) if wdtype == "bf16" else W_na.view(torch.int32),
                               W_ref.view(torch.int16) if wdtype == "bf16" else W_ref.view(torch.int32))
            assert torch.equal(state.view(torch.int32), ref.state.view(torch.int32))
            # diagnostics only: the oracle bar holds trivially once the bits agree
            check_state(state.cpu().numpy(), ref.state.cpu().numpy(), "state")
            check_weights(w_to_host(W_na), w_to_host(W_ref), 1e-3)
        assert ref.device_status() == 0
    finally:
        E.ember_destroy(h)
