"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Inputs come from the seeded presets; both sides read the same stored tensors.
Tolerances: routing bit-exact away from near-ties (margin < 1e-6 in log g);
combine weights rel. 2e-5; outputs rel. Frobenius 1e-4 (fp32) / 1e-2 (bf16)
and max abs 3e-2 (bf16).  Large presets are checked on a seeded sample of 256
token rows (tokens are independent in Eq. 1); their gate and routing are
checked on every token.
"""
import numpy as np
import pytest
import torch

from oracle import ec2moe_oracle as orc
from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import LayerRun, desc_for
from tests.parity import TIE_GAP, oracle_inputs, output_check, rel_fro, routing_check, weights_check

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()
    yield
    torch.cuda.synchronize()


def _np(t):
    return t.detach().to("cpu").to(torch.float64).numpy() if t.dtype.is_floating_point else t.detach().cpu().numpy()


def _gate_ref(cfg, inp):
    o = oracle_inputs({k: inp[k] for k in ("X", "W_local", "b_local", "W_global", "b_global", "mask")})
    return orc.gate_and_route(o["X"], o["W_local"], o["b_local"], o["W_global"], o["b_global"], o["mask"],
                              cfg.n_groups, cfg.k, bool(cfg.renorm_topk))


GATE_CASES = [
    S.preset("tiny_fp32"),
    S.preset("tiny_fp32", renorm_topk=1, seed=3),
    S.preset("switch_bf16"),
    S.preset("switch_bf16", T=1000, seed=1),
    S.preset("switch_bf16", T=1, seed=2),
    S.preset("mixtral_bf16"),
    S.preset("finegrained_bf16"),
    S.preset("finegrained_bf16", T=777, n_groups=4, seed=4, renorm_topk=1),
    S.preset("decode_bf16", T=1, n_allowed=4, seed=1),
    S.preset("decode_bf16", T=64, n_allowed=8, seed=64),
    S.preset("decode_bf16", T=256, n_allowed=4, seed=256),
    # every allowed expert selected (k = |E_local|); a whole group masked out
    S.preset("tiny_fp32", n_allowed=2, k=2, seed=5),
    S.preset("switch_bf16", T=513, E=16, n_groups=4, k=3, n_allowed=5, seed=6),
    # more token tiles than SMs (each CTA runs several tiles); d_model not a
    # multiple of the 64-column stage; exactly 80 gate rows; 136 gate rows
    S.preset("switch_bf16", T=20000, seed=17),
    S.preset("switch_bf16", T=300, d=200, seed=16),
    S.preset("finegrained_bf16", T=900, n_groups=16, k=4, seed=19),
    S.preset("finegrained_bf16", T=700, E=128, n_groups=8, n_allowed=64, k=4, seed=15),
    # d_model split over a two-CTA cluster per tile (d_model >= 2048): a
    # ragged last tile (104 rows, the second CTA owning rows 64..103), a
    # single tile with 6 rows in the second CTA's half, and the one-group
    # decision (K = 1, Top-2) over five tiles
    S.preset("mixtral_bf16", T=1000, seed=71),
    S.preset("mixtral_bf16", T=70, seed=72),
    S.preset("decode_bf16", T=600, n_allowed=6, seed=73),
]


@pytest.mark.parametrize("cfg", GATE_CASES, ids=lambda c: f"{c.name}-T{c.T}-K{c.n_groups}-k{c.k}-s{c.seed}")
def test_gate_topk(cfg):
    inp = S.make_inputs(cfg, device="cuda", with_experts=False)
    desc = desc_for(cfg)
    idx = torch.full((cfg.T, cfg.k), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    torch.cuda.synchronize()
    ref = _gate_ref(cfg, inp)
    gi, gw = idx.cpu().numpy(), w.cpu().numpy()
    n_cmp, n_excl = routing_check(gi, ref)
    # A token is excluded when its k-th and (k+1)-th choices are within 1e-6
    # in log g.  Those gaps have a density of order one near zero, so about
    # T * 1e-6 tokens (well below one at these sizes) are expected; the bound
    # leaves room for a few without hiding a systematic difference.
    assert n_excl <= max(2, cfg.T // 8192), n_excl
    weights_check(gi, gw, ref, ref["gap_boundary"] >= TIE_GAP)
    # masked experts never selected; counts over the kept tokens agree exactly
    mask = inp["mask"].cpu().numpy()
    assert mask[gi].all()
    keep = ref["gap_boundary"] >= TIE_GAP
    assert np.array_equal(np.bincount(gi[keep].ravel(), minlength=cfg.E),
                          np.bincount(ref["idx"][keep].ravel(), minlength=cfg.E))


NONFINITE_CASES = [S.preset("tiny_fp32", seed=21), S.preset("switch_bf16", T=300, seed=22),
                   S.preset("finegrained_bf16", T=300, seed=23),
                   S.preset("finegrained_bf16", T=300, E=128, n_groups=8, n_allowed=64, k=4, seed=24)]


@pytest.mark.parametrize("cfg", NONFINITE_CASES, ids=lambda c: f"{c.name}-E{c.E}")
def test_gate_nonfinite_token_names_valid_experts(cfg):
    """A token with NaN activations still gets k distinct allowed experts (the
    lowest allowed ones, with NaN weights); the other tokens are unaffected."""
    inp = S.make_inputs(cfg, device="cuda", with_experts=False)
    bad = [0, cfg.T // 2, cfg.T - 1]
    inp["X"][bad] = float("nan")
    desc = desc_for(cfg)
    idx = torch.full((cfg.T, cfg.k), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    torch.cuda.synchronize()
    gi, gw = idx.cpu().numpy(), w.cpu().numpy()
    allowed = np.flatnonzero(inp["mask"].cpu().numpy())
    for t in bad:
        assert sorted(gi[t].tolist()) == allowed[: cfg.k].tolist()
        assert np.isnan(gw[t]).all()
    good = np.setdiff1d(np.arange(cfg.T), bad)
    inp["X"][bad] = 0.0
    ref = _gate_ref(cfg, inp)
    sub = {key: (v[good] if isinstance(v, np.ndarray) and v.shape[:1] == (cfg.T,) else v) for key, v in ref.items()}
    n_cmp, n_excl = routing_check(gi[good], sub)
    assert n_excl <= 2, n_excl


@pytest.mark.parametrize("cfg", [S.preset("decode_bf16", T=16, n_allowed=4, seed=25),
                                 S.preset("finegrained_bf16", T=40, seed=26)], ids=lambda c: f"{c.name}-T{c.T}")
def test_layer_nonfinite_token_small_batch(cfg):
    """The small-batch gate of the layer path (d_model split across CTAs) takes
    the same decision for a NaN token: the k lowest allowed experts; its routing
    tables stay consistent."""
    inp = S.make_inputs(cfg, device="cuda")
    bad = [0, cfg.T - 1]
    inp["X"][bad] = float("nan")
    run = LayerRun(cfg, inp)
    run.forward()
    torch.cuda.synchronize()
    gi = run.topk_idx.cpu().numpy()
    allowed = np.flatnonzero(inp["mask"].cpu().numpy())
    for t in bad:
        assert sorted(gi[t].tolist()) == allowed[: cfg.k].tolist()
    assert np.array_equal(run.counts.cpu().numpy(), np.bincount(gi.ravel(), minlength=cfg.E))


ROUTE_CASES = [S.preset("tiny_fp32"), S.preset("switch_bf16"), S.preset("finegrained_bf16"),
               S.preset("switch_bf16", T=1000, k=2, seed=9), S.preset("decode_bf16", T=1, seed=1)]


@pytest.mark.parametrize("cfg", ROUTE_CASES, ids=lambda c: f"{c.name}-T{c.T}-k{c.k}")
def test_route_tables_and_gather(cfg):
    """Histogram / scan / permutation are integer functions of topk_idx: bit-exact."""
    inp = S.make_inputs(cfg, device="cuda", with_experts=False)
    desc = desc_for(cfg)
    n = cfg.T * cfg.k
    idx = torch.empty((cfg.T, cfg.k), dtype=torch.int32, device="cuda")
    w = torch.empty((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    counts = torch.full((cfg.E,), -1, dtype=torch.int32, device="cuda")
    offsets = torch.full((cfg.E + 1,), -1, dtype=torch.int32, device="cuda")
    perm = torch.full((n,), -1, dtype=torch.int32, device="cuda")
    inv = torch.full((n,), -1, dtype=torch.int32, device="cuda")
    dst = torch.empty((n, cfg.d), dtype=inp["X"].dtype, device="cuda")
    ws_b = C.ec2moe_route_workspace_size(desc)
    ws = torch.empty(max(ws_b, 16), dtype=torch.uint8, device="cuda")
    C.ec2moe_route(desc, idx, counts, offsets, perm, inv, inp["X"], cfg.d, dst, ws, ws_b)
    torch.cuda.synchronize()
    gi = idx.cpu().numpy()
    c_ref, o_ref, p_ref = orc.route_tables(gi, cfg.E)
    assert np.array_equal(counts.cpu().numpy(), c_ref)
    assert np.array_equal(offsets.cpu().numpy(), o_ref)
    assert np.array_equal(perm.cpu().numpy(), p_ref)
    pv = perm.cpu().numpy()
    assert np.array_equal(inv.cpu().numpy()[pv], np.arange(n))
    rows = torch.from_numpy((p_ref // cfg.k).astype(np.int64)).cuda()
    assert torch.equal(dst, inp["X"][rows])


CODEC_CASES = [S.preset("tiny_fp32"), S.preset("switch_bf16"), S.preset("switch_bf16", T=1000, seed=3),
               S.preset("mixtral_bf16"), S.preset("finegrained_bf16", T=4099, seed=2),
               S.preset("decode_bf16", T=4, r=128, seed=4)]


@pytest.mark.parametrize("cfg", CODEC_CASES, ids=lambda c: f"{c.name}-T{c.T}-r{c.r}")
def test_codec(cfg):
    g = S.make_generator(cfg.seed + 100, "cuda")
    dt = cfg.torch_dtype
    X = torch.randn(cfg.T, cfg.d, generator=g, device="cuda").to(dt)
    V_enc = (torch.randn(cfg.r, cfg.d, generator=g, device="cuda") / cfg.d ** 0.5).to(dt)
    V_dec = (torch.randn(cfg.d, cfg.r, generator=g, device="cuda") / cfg.r ** 0.5).to(dt)
    desc = desc_for(cfg)
    Z = torch.full((cfg.T, cfg.r), float("nan"), device="cuda").to(dt)
    Xh = torch.full((cfg.T, cfg.d), float("nan"), device="cuda").to(dt)
    C.ec2moe_lr_encode(desc, X, V_enc, Z)
    C.ec2moe_lr_decode(desc, Z, V_dec, Xh)
    torch.cuda.synchronize()
    bf = cfg.dtype == S.BF16
    Z_ref = orc.lr_encode(_np(X), _np(V_enc))
    output_check(_np(Z), Z_ref, bf)
    # the decoder is checked on the transmitted (stored) Z
    output_check(_np(Xh), orc.lr_decode(_np(Z), _np(V_dec)), bf)


LAYER_CASES = [
    (S.preset("tiny_fp32"), None),
    (S.preset("tiny_fp32", renorm_topk=1, k=1, n_groups=1, seed=7), None),
    (S.preset("switch_bf16"), None),
    (S.preset("switch_bf16", T=1000, k=2, n_groups=4, seed=8), None),
    (S.preset("switch_bf16", T=300, r=0, seed=9), None),
    (S.preset("switch_bf16", T=200, E=1, n_groups=1, n_allowed=1, k=1, seed=10), None),
    (S.preset("mixtral_bf16"), 256),
    (S.preset("switch_bf16", T=20000, seed=18), 256),
    (S.preset("finegrained_bf16"), 256),
    (S.preset("finegrained_bf16", T=999, r=0, seed=11), None),
    (S.preset("decode_bf16", T=1, n_allowed=4, r=128, seed=1), None),
    (S.preset("decode_bf16", T=16, n_allowed=8, r=256, seed=16), None),
    (S.preset("decode_bf16", T=256, n_allowed=4, r=512, seed=256), None),
    # decode-sized groups (the weight-streaming CUDA-core GEMM at <= 2 rows)
    (S.preset("decode_bf16", T=4, n_allowed=8, r=256, seed=41), None),
    (S.preset("finegrained_bf16", T=2, seed=42), None),
    (S.preset("switch_bf16", T=2, seed=43), None),
    (S.preset("decode_bf16", T=1, n_allowed=8, r=256, seed=46), None),
    (S.preset("mixtral_bf16", T=3, seed=44), None),
    # split-K reduce inside the swapped-operand down projection: all 16 entries
    # (T = 8, Top-2) and Top-3 with relative row placement
    (S.preset("decode_bf16", T=8, n_allowed=8, r=256, seed=61), None),
    (S.preset("decode_bf16", T=5, k=3, n_allowed=6, r=128, seed=62), None),
    # split-K encoder with a K range count the k-block count does not divide
    # (33 k-blocks of 64 in 11 ranges of 3)
    (S.preset("decode_bf16", T=7, d=2112, d_ff=2048, n_allowed=8, r=256, seed=49), None),
    # small batches with d_model split across the gate's CTAs: group gate
    # with several token tiles, 72 gate rows, and an fp32 layer
    (S.preset("mixtral_bf16", T=129, seed=50), None),
    (S.preset("finegrained_bf16", T=200, seed=51), None),
    (S.preset("finegrained_bf16", T=150, seed=63), None),
    (S.preset("tiny_fp32", T=100, d=1024, seed=52), None),
    (S.preset("tiny_fp32", T=7, seed=45), None),
    # the gate's two-CTA clusters with the fused row reservations: a last tile
    # of 44 tokens (the second CTA owns no token of it), and K = 1 over five
    # tiles
    (S.preset("mixtral_bf16", T=300, d_ff=1024, seed=74), None),
    (S.preset("decode_bf16", T=520, n_allowed=8, d_ff=1024, r=128, seed=75), None),
    # the limits: 128 experts in 16 groups, Top-8, 144 gate rows; and many
    # tiles per CTA in every kernel
    (S.preset("switch_bf16", T=1024, d=512, E=128, d_ff=512, n_groups=16, k=8, n_allowed=96, r=128, seed=47), 256),
    (S.preset("switch_bf16", T=65536, seed=48), 256),
]


@pytest.mark.parametrize("cfg,sample", LAYER_CASES,
                         ids=lambda v: (f"{v.name}-T{v.T}-E{v.E}-k{v.k}-r{v.r}-s{v.seed}" if hasattr(v, "name")
                                        else f"rows{v}"))
def test_layer_forward(cfg, sample):
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    run.forward()
    assert C.ec2moe_last_device_error() == C.OK
    torch.cuda.synchronize()
    o = oracle_inputs(inp, lazy_experts=True)
    rows = None
    if sample:
        rows = np.sort(np.random.default_rng(cfg.seed + 1).choice(cfg.T, sample, replace=False))
    ref = orc.layer_forward(o, cfg.n_groups, cfg.k, cfg.act, bool(cfg.renorm_topk), rows=rows)
    gi = run.topk_idx.cpu().numpy()
    routing_check(gi, ref)
    keep_all = ref["gap_boundary"] >= TIE_GAP
    weights_check(gi, run.topk_w.cpu().numpy(), ref, keep_all)
    assert np.array_equal(run.counts.cpu().numpy(), np.bincount(gi.ravel(), minlength=cfg.E))
    if keep_all.all():
        assert np.array_equal(run.counts.cpu().numpy(), ref["counts"])
    sel = ref["rows"]
    keep = keep_all[sel]
    y = _np(run.Y)[sel]
    output_check(y[keep], ref["y"][keep], cfg.dtype == S.BF16)
    if cfg.r > 0:
        Z = _np(run.Z)[sel]
        output_check(Z, ref["Z"], cfg.dtype == S.BF16)


@pytest.mark.parametrize("cfg", [S.preset("mixtral_bf16"), S.preset("finegrained_bf16"),
                                 S.preset("switch_bf16", T=65536, seed=48)], ids=lambda c: c.name + f"-T{c.T}")
def test_layer_sample_covers_a_partial_tail_tile(cfg):
    """At full size the output is checked on a sample of rows; this sample
    always holds every row of one expert group smaller than a 128-row m-tile,
    so a group whose only tile is partial (its tail) is checked whole.  The
    least-loaded allowed expert's local bias is lowered until it receives
    between 1 and 127 rows."""
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    run.forward()
    torch.cuda.synchronize()
    allowed = np.flatnonzero(inp["mask"].cpu().numpy())
    e = int(allowed[np.argmin(run.counts.cpu().numpy()[allowed])])
    base = float(inp["b_local"][e])
    for shift in (0.0, 1.0, 2.0, 3.0, 4.0, 5.0, 6.0, 8.0, 10.0, 13.0):
        inp["b_local"][e] = base - shift
        run.forward()
        torch.cuda.synchronize()
        c = int(run.counts[e])
        if 1 <= c <= 127:
            break
    assert 1 <= c <= 127, c
    assert C.ec2moe_last_device_error() == C.OK
    gi = run.topk_idx.cpu().numpy()
    group_rows = np.flatnonzero((gi == e).any(axis=1))
    rng = np.random.default_rng(cfg.seed + 7)
    rows = np.union1d(group_rows, rng.choice(cfg.T, 128, replace=False))
    ref = orc.layer_forward(oracle_inputs(inp, lazy_experts=True), cfg.n_groups, cfg.k, cfg.act,
                            bool(cfg.renorm_topk), rows=rows)
    routing_check(gi, ref)
    assert np.array_equal(run.counts.cpu().numpy(), np.bincount(gi.ravel(), minlength=cfg.E))
    keep = ref["gap_boundary"][rows] >= TIE_GAP
    assert keep[np.isin(rows, group_rows)].sum() >= len(group_rows) - 2
    output_check(_np(run.Y)[rows][keep], ref["y"][keep], True)


def test_layer_is_deterministic():
    cfg = S.preset("switch_bf16", T=1000, k=2, seed=12)
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    a = run.forward().clone()
    b = run.forward().clone()
    assert torch.equal(a, b)


def test_experts_and_combine_entry_points():
    """The unfused entry points chained by hand give the fused layer's output."""
    cfg = S.preset("finegrained_bf16", T=600, seed=13)
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    y_fused = run.forward().clone()
    desc = desc_for(cfg)
    T, k, d = cfg.T, cfg.k, cfg.d
    dt = cfg.torch_dtype
    idx = torch.empty((T, k), dtype=torch.int32, device="cuda")
    w = torch.empty((T, k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    Z = torch.empty((T, cfg.r), dtype=dt, device="cuda")
    Xh = torch.empty((T, d), dtype=dt, device="cuda")
    C.ec2moe_lr_encode(desc, inp["X"], inp["V_enc"], Z)
    C.ec2moe_lr_decode(desc, Z, inp["V_dec"], Xh)
    counts = torch.empty(cfg.E, dtype=torch.int32, device="cuda")
    offsets = torch.empty(cfg.E + 1, dtype=torch.int32, device="cuda")
    perm = torch.empty(T * k, dtype=torch.int32, device="cuda")
    Xp = torch.empty((T * k, d), dtype=dt, device="cuda")
    rws = C.ec2moe_route_workspace_size(desc)
    rw = torch.empty(max(rws, 16), dtype=torch.uint8, device="cuda")
    C.ec2moe_route(desc, idx, counts, offsets, perm, None, Xh, d, Xp, rw, rws)
    ews = C.ec2moe_experts_workspace_size(desc)
    ew = torch.empty(ews, dtype=torch.uint8, device="cuda")
    slot = torch.empty((T * k, d), dtype=dt, device="cuda")
    C.ec2moe_experts(desc, Xp, offsets, inp["W1"], inp["W3"], inp["W2"], w, perm, slot, ew, ews)
    shared = torch.empty((cfg.n_shared * T, d), dtype=dt, device="cuda")
    C.ec2moe_shared_experts(desc, Xh, inp["W1s"], inp["W3s"], inp["W2s"], shared, ew, ews)
    Y = torch.empty((T, d), dtype=dt, device="cuda")
    C.ec2moe_combine(desc, slot, shared, Y)
    torch.cuda.synchronize()
    assert torch.equal(Y, y_fused)
    assert torch.equal(idx, run.topk_idx)
    assert torch.equal(Z, run.Z)


def test_zero_token_experts_and_tail_tiles():
    """Experts that receive no token, and groups whose row count is not a tile multiple."""
    cfg = S.preset("switch_bf16", T=131, E=16, n_allowed=16, k=1, seed=14)
    inp = S.make_inputs(cfg, device="cuda")
    # push every token to experts 3 and 11 only
    inp["b_local"] = torch.full((16,), -30.0, device="cuda")
    inp["b_local"][3] = 0.0
    inp["b_local"][11] = 0.0
    run = LayerRun(cfg, inp)
    run.forward()
    torch.cuda.synchronize()
    counts = run.counts.cpu().numpy()
    assert counts.sum() == cfg.T and (counts[[3, 11]] > 0).all() and counts[np.r_[0:3, 4:11, 12:16]].sum() == 0
    ref = orc.layer_forward(oracle_inputs(inp), cfg.n_groups, cfg.k, cfg.act)
    keep = ref["gap_boundary"] >= TIE_GAP
    output_check(_np(run.Y)[keep], ref["y"][keep], True)
