"""Exact ties in the gate: the lower expert index takes the earlier slot.

Two experts get bitwise-identical gate rows and biases ("twins"), either inside
one group, or across two groups that are identical copies of each other (same
local rows, same global row and bias, same mask pattern), so the fused score
log p_group + log p_local of each twin pair is computed from the same fp32
operands in the same order and ties exactly.  The expected routing is the
oracle's Top-k with each twin's g set to its partner's (the two are equal by
construction), which the stable sort resolves to the lower index; it is
compared bit for bit with no near-tie exclusion for the designed ties.  Tokens
excluded are only those with an accidental near-tie (< 1e-6 in log g) between
two experts that are not twins; the test also checks that the designed ties
decide many tokens.  Both ec2moe_gate and the layer call are checked, on the
tensor-core gate (bf16; two CTAs per tile at d_model >= 2048), the
small-batch split-d gate (<= 256 tokens, d_model >= 1024) and the SIMT gate
(fp32).  Twin experts also get identical
expert weights, so the layer's output is checked against the oracle whichever
twin each side picks.
"""
import numpy as np
import pytest
import torch

from oracle import ec2moe_oracle as orc
from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import LayerRun, desc_for
from tests.parity import TIE_GAP, oracle_inputs, output_check

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()
    yield
    torch.cuda.synchronize()


def _twin_inputs(cfg, mode):
    """Inputs with designed twins.  mode 'group': experts (1, E-2) share one
    group (K = 1) and are boosted so they usually both make the top-k.
    mode 'groups': groups 0 and 1 are copies; expert i of group 0 twins with
    expert i + E/K of group 1."""
    inp = S.make_inputs(cfg, device="cuda")
    E, K = cfg.E, cfg.n_groups
    mask = torch.ones(E, dtype=torch.uint8, device="cuda")
    if mode == "group":
        twins = [(1, E - 2)]
        src, dst = [1], [E - 2]
        inp["b_local"][1] = 2.0
        mask[0] = 0  # a masked expert as well
    else:
        M = E // K
        twins = [(i, i + M) for i in range(M)]
        src, dst = list(range(M)), list(range(M, 2 * M))
        mask[M - 1] = 0
        mask[2 * M - 1] = 0
        inp["W_global"][1] = inp["W_global"][0]
        inp["b_global"][0] = 2.5  # the twin groups win most tokens
        inp["b_global"][1] = 2.5
        if K > 2:
            mask[2 * M:3 * M] = 0  # plus a dead group
    for s_, d_ in zip(src, dst):
        inp["W_local"][d_] = inp["W_local"][s_]
        inp["b_local"][d_] = inp["b_local"][s_]
        for key in ("W1", "W3", "W2"):
            if inp.get(key) is not None:
                inp[key][d_] = inp[key][s_]
    inp["mask"] = mask
    return inp, twins


def _expected(cfg, inp, twins):
    """Oracle routing with every twin's g set to its partner's; returns
    (expected idx, keep mask, number of tokens a designed tie decides)."""
    o = oracle_inputs({k: inp[k] for k in ("X", "W_local", "b_local", "W_global", "b_global", "mask")})
    ref = orc.gate_and_route(o["X"], o["W_local"], o["b_local"], o["W_global"], o["b_global"], o["mask"],
                             cfg.n_groups, cfg.k, bool(cfg.renorm_topk))
    g, log_g = ref["g"].copy(), ref["log_g"].copy()
    for a, b in twins:
        g[:, b] = g[:, a]
        log_g[:, b] = log_g[:, a]
    allowed = ref["allowed"]
    idx = orc.topk_route(g, allowed, cfg.k)
    twin_of = {}
    for a, b in twins:
        twin_of[a], twin_of[b] = b, a
    order = np.argsort(np.where(allowed[None, :], -log_g, np.inf), axis=1, kind="stable")
    depth = min(cfg.k + 1, int(allowed.sum()))
    keep = np.ones(cfg.T, dtype=bool)
    decided = 0
    for t in range(cfg.T):
        top = order[t, :depth]
        tie_here = False
        for j in range(depth - 1):
            a, b = int(top[j]), int(top[j + 1])
            gap = log_g[t, a] - log_g[t, b]
            if twin_of.get(a) == b:
                tie_here = True
            elif gap < TIE_GAP:
                keep[t] = False
        decided += tie_here and keep[t]
    return idx, keep, decided, ref


TIE_CASES = [
    (S.preset("switch_bf16", T=1000, k=2, n_groups=1, seed=61), "group"),
    (S.preset("switch_bf16", T=1000, k=1, n_groups=1, seed=62), "group"),
    (S.preset("switch_bf16", T=777, E=16, k=3, n_groups=4, seed=63), "groups"),
    (S.preset("finegrained_bf16", T=600, seed=64), "groups"),
    (S.preset("mixtral_bf16", T=129, d_ff=1024, seed=65), "groups"),
    (S.preset("mixtral_bf16", T=400, d_ff=1024, seed=67), "groups"),
    (S.preset("tiny_fp32", T=200, seed=66), "groups"),
]


@pytest.mark.parametrize("cfg,mode", TIE_CASES,
                         ids=lambda v: f"{v.name}-T{v.T}-K{v.n_groups}-k{v.k}" if hasattr(v, "name") else v)
def test_exact_ties_go_to_the_lower_index(cfg, mode):
    inp, twins = _twin_inputs(cfg, mode)
    exp_idx, keep, decided, ref = _expected(cfg, inp, twins)
    assert decided >= cfg.T // 4, f"designed ties decide only {decided} tokens"
    assert (~keep).sum() <= 2, f"{(~keep).sum()} accidental near-ties"
    # the standalone gate
    desc = desc_for(cfg)
    idx = torch.full((cfg.T, cfg.k), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    torch.cuda.synchronize()
    gi = idx.cpu().numpy()
    bad = np.flatnonzero((gi != exp_idx).any(axis=1) & keep)
    assert bad.size == 0, f"gate: t={bad[:4]} got {gi[bad[:1]]} expected {exp_idx[bad[:1]]}"
    # the layer call (its own gate kernels, fused routing, experts)
    run = LayerRun(cfg, inp)
    run.forward()
    assert C.ec2moe_last_device_error() == C.OK
    torch.cuda.synchronize()
    li = run.topk_idx.cpu().numpy()
    bad = np.flatnonzero((li != exp_idx).any(axis=1) & keep)
    assert bad.size == 0, f"layer: t={bad[:4]} got {li[bad[:1]]} expected {exp_idx[bad[:1]]}"
    counts = run.counts.cpu().numpy()
    assert np.array_equal(counts, np.bincount(li.ravel(), minlength=cfg.E))
    if keep.all():
        assert np.array_equal(counts, np.bincount(exp_idx.ravel(), minlength=cfg.E))
    # the output: twins have identical experts, so y does not depend on the pick
    o = oracle_inputs(inp, lazy_experts=True)
    y_ref = orc.layer_forward(o, cfg.n_groups, cfg.k, cfg.act, bool(cfg.renorm_topk))["y"]
    y = run.Y.detach().to("cpu", torch.float64).numpy()
    output_check(y[keep], y_ref[keep], cfg.dtype == S.BF16)
