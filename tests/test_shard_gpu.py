"""Row-sharded dense step on one GPU: nshards emulated ranks, each with its
own handle, state and rows of W and G, run ember_shard_reduce, exchange
their blocks (a concatenation in shard order, what an all-gather gives),
then ember_shard_update.  W, r and c must be bit-identical to
ember_step_dense on the whole table, for every shard count (Section 2.3:
the statistics are sums of g^2 and the result is bitwise identical however
the rows are spread).  No kernel waits on another: the ranks run one after
the other.
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


def run_sharded(V, D, wdtype, opt, nshards, steps, dev):
    ref = make(V, D, wdtype, opt)
    W0 = (torch.randn(V, D, generator=torch.Generator(device=dev).manual_seed(7), device=dev) * 0.02).to(
        torch.bfloat16 if wdtype == "bf16" else torch.float32)
    Wref = W0.clone()
    ranks = [make(V, D, wdtype, opt) for _ in range(nshards)]
    plan = [ranks[k].shard_rows(k, nshards) for k in range(nshards)]
    nbytes = ranks[0].shard_exchange_bytes(nshards)
    Ws = [W0[r0:r0 + n].clone() for r0, n in plan]
    blocks = [torch.zeros(nbytes, dtype=torch.uint8, device=dev) for _ in range(nshards)]
    for t in range(1, steps + 1):
        G = grad(V, D, t, dev)
        ref.step_dense(Wref, G, 1e-3, t)
        Gs = [G[r0:r0 + n].contiguous() for r0, n in plan]
        for k in range(nshards):
            ranks[k].shard_reduce(k, nshards, Gs[k], blocks[k])
        gathered = torch.cat(blocks)
        for k in range(nshards):
            ranks[k].shard_update(k, nshards, Ws[k], Gs[k], gathered, 1e-3, t)
    torch.cuda.synchronize()
    return ref, Wref, ranks, plan, Ws


def bits(x):
    return x.view(torch.int16) if x.dtype == torch.bfloat16 else x.view(torch.int32)


@pytest.mark.parametrize("V,D", [(1000, 200), (3001, 256), (305, 132), (40, 8192), (777, 1028), (5, 7)])
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
    """V = 300 rows: 300 CTAs; 305 shards leave the last five empty, whose
    calls still keep c."""
    ref, Wref, ranks, plan, Ws = run_sharded(300, 64, "bf16", Opt(), 305, 2, cuda_device)
    assert [n for _, n in plan[-5:]] == [0] * 5
    assert torch.equal(bits(torch.cat(Ws)), bits(Wref))
    assert torch.equal(bits(ranks[-1].c), bits(ref.c))


def test_sharded_row_variant_is_refused(cuda_device):
    emb = Ember(100, 64, variant="row")
    blk = torch.zeros(emb.shard_exchange_bytes(2), dtype=torch.uint8, device=cuda_device)
    G = torch.zeros(50, 64, device=cuda_device)
    with pytest.raises(EmberError) as ex:
        emb.shard_reduce(0, 2, G, blk)
    assert ex.value.status == EMBER_ERR_UNSUPPORTED
