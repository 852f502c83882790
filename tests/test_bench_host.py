"""Host-side logic of bench.py, on the CPU: the algorithmic byte counts the
GB/s figures divide by, and which timed steps record kernel boundaries.

The byte counts follow from what Algorithm 1 forces (Section 2.3: the
update needs column statistics of every row, so G is read twice unless it
stays on chip): 4VD for the reduction read, 4VD + 2wVD for the apply pass
(G read again, W read and written), 8(V + D) for the state.
"""
import pytest

import bench
from paper_2607_01455_gb300 import synth


@pytest.mark.parametrize("name,gb", [
    ("dense_v32000_d4096_bf16", 1.573), ("dense_tied_v151936_d896_bf16", 1.635),
    ("dense_lmhead_v128256_d8192_bf16", 12.61), ("dense_wide_v128256_d16384_bf16", 25.22),
])
def test_dense_step_bytes(name, gb):
    wl = synth.WORKLOADS[name]
    assert bench.step_bytes(wl) / 1e9 == pytest.approx(gb, rel=2e-3)


def test_dense_step_bytes_small_fp32_table():
    """16VD + 8(V + D) for fp32 W: 1,057,280 bytes at 1024 x 64."""
    assert bench.step_bytes(synth.WORKLOADS["dense_v1024_d64_f32"]) == 16 * 1024 * 64 + 8 * (1024 + 64)


@pytest.mark.parametrize("name", ["dense_v32000_d4096_bf16", "dense_lmhead_v128256_d8192_bf16",
                                  "dense_v1024_d64_f32"])
def test_kernel_bytes_add_up_to_the_step(name):
    """The three kernels carry the step's bytes plus the apply pass's second
    read of r and c, 4(V + D): the step counts the state read and written
    once."""
    wl = synth.WORKLOADS[name]
    kb = bench.kernel_bytes(wl)
    assert kb["reduce"] + kb["apply"] + kb["state"] == bench.step_bytes(wl) + 4 * (wl.V + wl.D)
    w = 2 if wl.wdtype == "bf16" else 4
    assert kb["apply"] == (4 + 2 * w) * wl.V * wl.D + 4 * (wl.V + wl.D)


def test_sparse_step_bytes():
    """With U = 8681 distinct ids among N = 32768: 0.484 GB per step."""
    wl = synth.WORKLOADS["sparse_v262144_d2048_bf16_n32768"]
    assert bench.sparse_bytes(wl, 8681) == 484155392
    # per distinct id: its summed row written and read (8D) and its W row
    # read and written (4D, bf16) ...
    base = bench.sparse_bytes(wl, 0)
    assert bench.sparse_bytes(wl, 100) - base == 100 * 12 * wl.D
    # ... until re-reading the N occurrence rows (4ND) is the cheaper
    # second visit
    assert bench.sparse_bytes(wl, wl.N) - base == 4 * wl.N * wl.D + 4 * wl.N * wl.D


@pytest.mark.parametrize("steps", [2, 3, 4, 5, 8, 400])
def test_traced_steps_leave_untraced_ones(steps):
    t = bench.traced_steps(steps)
    assert t and len(t) < steps
    assert all(0 <= k < steps for k in t)
    if steps >= bench.TRACE_EVERY:
        assert t == list(range(bench.TRACE_EVERY - 1, steps, bench.TRACE_EVERY))


def test_traced_steps_refuse_a_single_step():
    with pytest.raises(SystemExit):
        bench.traced_steps(1)
