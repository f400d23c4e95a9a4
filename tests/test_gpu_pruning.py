"""Top-group pruning of the group gate through the C ABI, against the oracle's
group_gate_pruned (Eq. 6 first, the top groups by p_group kept, Eq. 5 inside
them, Eq. 7 with p_group renormalised over the kept groups).

Routing is bit-exact away from near-ties; with pruning the margin also covers
the group decision (the gap in m between the last kept and the best pruned
group).  Cases cover the tensor-core gate (bf16), the small-batch split-d gate
(<= 256 tokens, d_model >= 1024), the SIMT gate (fp32), a dead group, and
top_groups at and above the number of live groups (no pruning).
"""
import numpy as np
import pytest
import torch

from oracle import ec2moe_oracle as orc
from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import LayerRun, desc_for
from tests.parity import TIE_GAP, oracle_inputs, output_check, routing_check, weights_check

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()
    yield
    torch.cuda.synchronize()


def _ref(cfg, inp):
    o = oracle_inputs({k: inp[k] for k in ("X", "W_local", "b_local", "W_global", "b_global", "mask")})
    return orc.gate_and_route(o["X"], o["W_local"], o["b_local"], o["W_global"], o["b_global"], o["mask"],
                              cfg.n_groups, cfg.k, bool(cfg.renorm_topk), top_groups=cfg.top_groups)


PRUNE_CASES = [
    S.preset("switch_bf16", T=1000, E=16, n_groups=4, k=2, n_allowed=12, top_groups=2, seed=71),
    S.preset("switch_bf16", T=513, E=16, n_groups=4, k=1, n_allowed=16, top_groups=1, seed=72),
    S.preset("finegrained_bf16", T=777, top_groups=3, seed=73),
    S.preset("finegrained_bf16", T=600, top_groups=3, k=4, renorm_topk=1, seed=74),
    S.preset("mixtral_bf16", T=129, d_ff=1024, top_groups=1, n_allowed=8, seed=75),
    S.preset("mixtral_bf16", T=300, d_ff=1024, top_groups=1, n_allowed=8, seed=79),
    S.preset("tiny_fp32", T=256, n_allowed=8, top_groups=1, seed=76),
    S.preset("switch_bf16", T=300, E=16, n_groups=4, k=2, n_allowed=16, top_groups=4, seed=77),
]


def _inputs(cfg):
    inp = S.make_inputs(cfg, device="cuda")
    if cfg.n_groups > 1:
        # spread the group logits so that pruning changes many routings
        inp["b_global"].copy_(torch.linspace(0.6, -0.6, cfg.n_groups, device="cuda"))
    return inp


@pytest.mark.parametrize("cfg", PRUNE_CASES, ids=lambda c: f"{c.name}-T{c.T}-K{c.n_groups}-G{c.top_groups}-k{c.k}")
def test_pruned_gate(cfg):
    inp = _inputs(cfg)
    ref = _ref(cfg, inp)
    desc = desc_for(cfg)
    idx = torch.full((cfg.T, cfg.k), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    torch.cuda.synchronize()
    gi, gw = idx.cpu().numpy(), w.cpu().numpy()
    n_cmp, n_excl = routing_check(gi, ref)
    assert n_excl <= 2, n_excl
    keep = ref["gap_boundary"] >= TIE_GAP
    weights_check(gi, gw, ref, keep)
    # pruning must matter for these inputs (unless nothing is pruned)
    full = orc.gate_and_route(*[S.to_f64(inp[k]) if inp[k] is not None else None
                                for k in ("X", "W_local", "b_local", "W_global", "b_global")],
                              inp["mask"].cpu().numpy(), cfg.n_groups, cfg.k, bool(cfg.renorm_topk))
    live = sum(inp["mask"].cpu().numpy().reshape(cfg.n_groups, -1).any(axis=1))
    changed = int((full["idx"] != ref["idx"]).any(axis=1).sum())
    if cfg.top_groups < live:
        assert changed > cfg.T // 20, changed
    else:
        assert changed == 0


@pytest.mark.parametrize("cfg", [PRUNE_CASES[0], PRUNE_CASES[2], PRUNE_CASES[4], PRUNE_CASES[5]],
                         ids=lambda c: f"{c.name}-T{c.T}-G{c.top_groups}")
def test_pruned_layer(cfg):
    inp = _inputs(cfg)
    run = LayerRun(cfg, inp)
    run.forward()
    assert C.ec2moe_last_device_error() == C.OK
    torch.cuda.synchronize()
    o = oracle_inputs(inp, lazy_experts=True)
    rows = None
    if cfg.d * cfg.d_ff > 768 * 3072:
        rows = np.sort(np.random.default_rng(cfg.seed).choice(cfg.T, min(cfg.T, 128), replace=False))
    ref = orc.layer_forward(o, cfg.n_groups, cfg.k, cfg.act, bool(cfg.renorm_topk), rows=rows,
                            top_groups=cfg.top_groups)
    gi = run.topk_idx.cpu().numpy()
    routing_check(gi, ref)
    keep_all = ref["gap_boundary"] >= TIE_GAP
    weights_check(gi, run.topk_w.cpu().numpy(), ref, keep_all)
    assert np.array_equal(run.counts.cpu().numpy(), np.bincount(gi.ravel(), minlength=cfg.E))
    sel = ref["rows"]
    keep = keep_all[sel]
    y = run.Y.detach().to("cpu", torch.float64).numpy()[sel]
    output_check(y[keep], ref["y"][keep], cfg.dtype == S.BF16)


def test_pruned_dead_group_and_rejection():
    # group 0 has no allowed expert; keeping 1 of the 3 live groups
    cfg = S.preset("switch_bf16", T=400, E=16, n_groups=4, k=2, n_allowed=16, top_groups=1, seed=78)
    inp = _inputs(cfg)
    inp["mask"] = torch.tensor([0, 0, 0, 0] + [1] * 12, dtype=torch.uint8, device="cuda")
    ref = _ref(cfg, inp)
    desc = desc_for(cfg)
    idx = torch.full((cfg.T, cfg.k), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    torch.cuda.synchronize()
    gi = idx.cpu().numpy()
    routing_check(gi, ref)
    assert (gi >= 4).all()
    # every routed pair of a token lies in one group (one group kept)
    assert ((gi[:, 0] // 4) == (gi[:, 1] // 4)).all()
    # a group that holds a single allowed expert makes Top-2 impossible under G = 1
    inp["mask"] = torch.tensor([1, 0, 0, 0] + [1] * 12, dtype=torch.uint8, device="cuda")
    with pytest.raises(C.Ec2moeError) as e:
        C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                      inp["mask"].cpu(), idx, w)
    assert e.value.status == C.ERR_TOO_FEW_EXPERTS
