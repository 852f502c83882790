"""Row-sharded dense step on one GPU: nshards emulated ranks, each with its
own handle, state and rows of W and G, run ember_shard_reduce, combine their
exponent blocks with an elementwise max (what an all-reduce MAX gives), run
ember_shard_pack, add their fixed-point blocks (an all-reduce SUM), then run
ember_shard_update.  W, r and c must be bit-identical to ember_step_dense on
the whole table, for every shard count (Section 2.3: the statistics are sums
of g^2 and the result is bitwise identical however the rows are spread).  No
kernel waits on another: the ranks run one after the other.
"""
import pytest
import torch

from paper_2607_01455_gb300.ember import Ember, EmberError, EMBER_ERR_UNSUPPORTED
from parity import Opt

pytestmark = pytest.mark.gpu


def make(V, D, wdtype, opt):
    return Ember(V, D, wdtype=wdtype, beta2=opt.beta2, eps=opt.eps, maximize=opt.maximize,
                 bias_correction=opt.bias_correction, variant=opt.variant)


def grad(V, D, t, dev):
    g = torch.Generator(device=dev).manual_seed(1000 + t)
    G = torch.randn(V, D, generator=g, device=dev) * 1e-3
    G *= torch.rand(V, 1, generator=g, device=dev) * 2 + 0.01
    return G


def sharded_step(ranks, plan, Ws, Gs, lr, t, dev):
    """One step of the three-call protocol over emulated ranks; returns the
    all-reduced blocks."""
    n = len(ranks)
    D = ranks[0].D
    scales = [torch.zeros(D + 1, dtype=torch.uint8, device=dev) for _ in range(n)]
    for k in range(n):
        ranks[k].shard_reduce(k, n, Gs[k], scales[k])
    smax = torch.stack(scales).amax(0)  # all-reduce MAX
    sums = [torch.zeros(D + 1, dtype=torch.int64, device=dev) for _ in range(n)]
    for k in range(n):
        ranks[k].shard_pack(k, n, smax, sums[k])
    ssum = torch.stack(sums).sum(0)  # all-reduce SUM (the totals stay below 2^63)
    for k in range(n):
        ranks[k].shard_update(k, n, Ws[k], Gs[k], smax, ssum, lr, t)
    return smax, ssum


def run_sharded(V, D, wdtype, opt, nshards, steps, dev):
    ref = make(V, D, wdtype, opt)
    W0 = (torch.randn(V, D, generator=torch.Generator(device=dev).manual_seed(7), device=dev) * 0.02).to(
        torch.bfloat16 if wdtype == "bf16" else torch.float32)
    Wref = W0.clone()
    ranks = [make(V, D, wdtype, opt) for _ in range(nshards)]
    plan = [ranks[k].shard_rows(k, nshards) for k in range(nshards)]
    Ws = [W0[r0:r0 + n].clone() for r0, n in plan]
    for t in range(1, steps + 1):
        G = grad(V, D, t, dev)
        ref.step_dense(Wref, G, 1e-3, t)
        Gs = [G[r0:r0 + n].contiguous() for r0, n in plan]
        sharded_step(ranks, plan, Ws, Gs, 1e-3, t, dev)
    torch.cuda.synchronize()
    return ref, Wref, ranks, plan, Ws


def bits(x):
    return x.view(torch.int16) if x.dtype == torch.bfloat16 else x.view(torch.int32)


@pytest.mark.parametrize("V,D", [(1000, 200), (3001, 256), (305, 132), (40, 8192), (777, 1028), (5, 7),
                                 (32000, 1024)])
@pytest.mark.parametrize("nshards", [1, 2, 3, 4, 8])
def test_sharded_step_is_bitwise_the_whole_table_step(cuda_device, V, D, nshards):
    ref, Wref, ranks, plan, Ws = run_sharded(V, D, "bf16", Opt(), nshards, 3, cuda_device)
    assert torch.equal(bits(torch.cat(Ws)), bits(Wref))
    for k, (r0, n) in enumerate(plan):
        assert torch.equal(bits(ranks[k].r[r0:r0 + n]), bits(ref.r[r0:r0 + n]))
        assert torch.equal(bits(ranks[k].c), bits(ref.c))
        assert ranks[k].device_status() == 0


@pytest.mark.parametrize("opt", [Opt(variant="col"), Opt(maximize=True), Opt(bias_correction=False),
                                 Opt(beta2=0.9, eps=1e-6)],
                         ids=["col", "maximize", "no-bias-correction", "beta2-0.9"])
def test_sharded_step_hyperparameters_fp32(cuda_device, opt):
    V, D = 1000, 200
    ref, Wref, ranks, plan, Ws = run_sharded(V, D, "f32", opt, 3, 3, cuda_device)
    assert torch.equal(bits(torch.cat(Ws)), bits(Wref))
    for k, (r0, n) in enumerate(plan):
        assert torch.equal(bits(ranks[k].c), bits(ref.c))


def test_more_shards_than_ctas(cuda_device):
    """V = 300 rows, D = 2048: 300 CTAs; 305 shards leave the last five empty,
    whose calls still take part and keep c."""
    ref, Wref, ranks, plan, Ws = run_sharded(300, 2048, "bf16", Opt(), 305, 2, cuda_device)
    assert [n for _, n in plan[-5:]] == [0] * 5
    assert torch.equal(bits(torch.cat(Ws)), bits(Wref))
    assert torch.equal(bits(ranks[-1].c), bits(ref.c))


def test_columns_of_very_different_scales(cuda_device):
    """Each column's exponent is negotiated on its own: columns whose sums of
    g^2 differ by 2^120 keep their full precision and the sharded step stays
    bitwise the whole-table step."""
    V, D = 2000, 64
    dev = cuda_device
    ref = make(V, D, "f32", Opt())
    ranks = [make(V, D, "f32", Opt()) for _ in range(4)]
    plan = [ranks[k].shard_rows(k, 4) for k in range(4)]
    W0 = torch.randn(V, D, generator=torch.Generator(device=dev).manual_seed(3), device=dev) * 0.02
    Wref = W0.clone()
    Ws = [W0[r0:r0 + n].clone() for r0, n in plan]
    scale = torch.pow(2.0, torch.linspace(-30, 30, D, device=dev))
    for t in (1, 2):
        G = grad(V, D, t, dev) * scale
        ref.step_dense(Wref, G, 1e-3, t)
        Gs = [G[r0:r0 + n].contiguous() for r0, n in plan]
        sharded_step(ranks, plan, Ws, Gs, 1e-3, t, dev)
    torch.cuda.synchronize()
    assert torch.equal(bits(torch.cat(Ws)), bits(Wref))
    assert torch.equal(bits(ranks[0].c), bits(ref.c))
    # c is the EMA of the column means of g^2 to fp32 precision at every scale
    G1, G2 = grad(V, D, 1, dev).double() * scale.double(), grad(V, D, 2, dev).double() * scale.double()
    c_exact = 0.999 * (0.001 * (G1 ** 2).mean(0)) + 0.001 * (G2 ** 2).mean(0)
    rel = ((ref.c.double() - c_exact).abs() / c_exact).max().item()
    assert rel < 1e-5, rel


def test_sharded_row_variant_is_refused(cuda_device):
    emb = Ember(100, 64, variant="row")
    blk = torch.zeros(emb.shard_scale_bytes(), dtype=torch.uint8, device=cuda_device)
    G = torch.zeros(50, 64, device=cuda_device)
    with pytest.raises(EmberError) as ex:
        emb.shard_reduce(0, 2, G, blk)
    assert ex.value.status == EMBER_ERR_UNSUPPORTED
