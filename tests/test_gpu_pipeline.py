"""The end/cloud pipelined layer call (two streams, micro-batches) through the
C ABI: same routing, histogram, transmitted Z and output as the one-stream
layer call, and parity with the oracle (the pipelined output of every case is
held to the oracle's tolerances, not only to the one-stream call's)."""
import numpy as np
import pytest
import torch

from oracle import ec2moe_oracle as orc
from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import LayerRun
from tests.parity import TIE_GAP, oracle_inputs, output_check, routing_check, weights_check

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()
    yield
    torch.cuda.synchronize()


def _pipelined(run, n_micro, same_stream=False):
    cur = torch.cuda.current_stream()
    s_end = torch.cuda.Stream()
    s_cloud = s_end if same_stream else torch.cuda.Stream()
    s_end.wait_stream(cur)
    run.Y.fill_(float("nan"))
    run.topk_idx.fill_(-1)
    run.counts.fill_(-1)
    run.forward_pipelined(n_micro, s_end, s_cloud)
    cur.wait_stream(s_end)
    torch.cuda.synchronize()
    assert C.ec2moe_last_device_error() == C.OK
    return (run.Y.clone(), run.topk_idx.clone(), run.topk_w.clone(), run.counts.clone(),
            None if run.Z is None else run.Z.clone())


PIPE_CASES = [
    (S.preset("switch_bf16", T=1000, seed=31), 3),
    (S.preset("switch_bf16", T=1000, k=2, n_groups=4, seed=37), 5),
    (S.preset("finegrained_bf16", T=777, seed=32), 4),
    (S.preset("mixtral_bf16", T=600, seed=35), 2),
    (S.preset("switch_bf16", T=300, r=0, seed=34), 2),
    (S.preset("tiny_fp32", seed=33), 2),
    (S.preset("decode_bf16", T=5, n_allowed=8, seed=36), 8),
    (S.preset("decode_bf16", T=300, n_allowed=8, r=128, seed=39), 2),
    (S.preset("switch_bf16", T=4096), 1),
]


@pytest.mark.parametrize("cfg,n_micro", PIPE_CASES,
                         ids=lambda v: f"{v.name}-T{v.T}-k{v.k}-r{v.r}" if hasattr(v, "name") else f"m{v}")
def test_pipelined_matches_one_stream_layer(cfg, n_micro):
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    run.forward()
    torch.cuda.synchronize()
    ref = (run.Y.clone(), run.topk_idx.clone(), run.topk_w.clone(), run.counts.clone(),
           None if run.Z is None else run.Z.clone())
    # The layer's gate splits d_model across CTAs for batches of <= 256 tokens
    # (d_model >= 1024), and the encoder splits its K range for batches of
    # <= 256 rows in a number of ranges set by the 128-row tiles: the batch and
    # its micro-batches take the same gate / encoder when they fall in the
    # same class, else results agree up to rounding.
    sub = -(-cfg.T // n_micro)
    small_gate = lambda t: t <= 256 and cfg.d >= 1024
    same_gate = small_gate(cfg.T) == small_gate(sub)
    same_z = cfg.r == 0 or (cfg.T > 256 and sub > 256) or (cfg.T <= 128 and sub <= 128)
    ref_gate = None if same_gate else _gate_ref(cfg, inp)
    # the oracle, for the pipelined output itself (a seeded sample of rows on
    # the large-expert shape)
    rows = None
    if cfg.d * cfg.d_ff > 768 * 3072:
        rows = np.sort(np.random.default_rng(cfg.seed).choice(cfg.T, min(cfg.T, 128), replace=False))
    ref_layer = orc.layer_forward(oracle_inputs(inp, lazy_experts=True), cfg.n_groups, cfg.k, cfg.act,
                                  bool(cfg.renorm_topk), rows=rows)
    for same in (False, True):
        got = _pipelined(run, n_micro, same_stream=same)
        gi = got[1].cpu().numpy()
        routing_check(gi, ref_layer)
        sel = ref_layer["rows"]
        keep_o = ref_layer["gap_boundary"][sel] >= TIE_GAP
        output_check(got[0].to("cpu", torch.float64).numpy()[sel][keep_o], ref_layer["y"][keep_o],
                     cfg.dtype == S.BF16)
        if same_gate:
            assert torch.equal(got[1], ref[1]) and torch.equal(got[2], ref[2]) and torch.equal(got[3], ref[3])
            rows = slice(None)
        else:
            # both gates against the oracle; outputs compared where they agree
            keep = ref_gate["gap_boundary"] >= TIE_GAP
            for r in (got, ref):
                gi = r[1].cpu().numpy()
                routing_check(gi, ref_gate)
                weights_check(gi, r[2].cpu().numpy(), ref_gate, keep)
                assert np.array_equal(r[3].cpu().numpy(), np.bincount(gi.ravel(), minlength=cfg.E))
            rows = (got[1] == ref[1]).all(dim=1).cpu().numpy()
        if ref[4] is not None:
            if same_z:
                assert torch.equal(got[4], ref[4])
            else:
                output_check(got[4].to("cpu", torch.float64).numpy(), ref[4].to("cpu", torch.float64).numpy(),
                             cfg.dtype == S.BF16, pair=True)
        if same_gate and same_z and (cfg.T * cfg.k <= 2 or sub * cfg.k > 2):
            assert torch.equal(got[0], ref[0])  # the same kernels on both sides
        else:
            # micro-batches of <= 2 rows per expert take the weight-streaming
            # GEMM, the whole batch the tensor-core one (or the gates or the
            # encoders differ, above): equal up to rounding
            output_check(got[0].to("cpu", torch.float64).numpy()[rows], ref[0].to("cpu", torch.float64).numpy()[rows],
                         cfg.dtype == S.BF16, pair=True)


def _gate_ref(cfg, inp):
    o = oracle_inputs({k: inp[k] for k in ("X", "W_local", "b_local", "W_global", "b_global", "mask")})
    return orc.gate_and_route(o["X"], o["W_local"], o["b_local"], o["W_global"], o["b_global"], o["mask"],
                              cfg.n_groups, cfg.k, bool(cfg.renorm_topk))


def test_pipelined_parity_with_oracle():
    cfg = S.preset("finegrained_bf16", T=513, seed=38)
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    Y, idx, w, counts, Z = _pipelined(run, 3)
    o = oracle_inputs(inp, lazy_experts=True)
    ref = orc.layer_forward(o, cfg.n_groups, cfg.k, cfg.act, bool(cfg.renorm_topk))
    gi = idx.cpu().numpy()
    routing_check(gi, ref)
    keep = ref["gap_boundary"] >= TIE_GAP
    assert np.array_equal(counts.cpu().numpy(), np.bincount(gi.ravel(), minlength=cfg.E))
    y = Y.detach().to("cpu", torch.float64).numpy()
    output_check(y[keep], ref["y"][keep], True)
    output_check(Z.detach().to("cpu", torch.float64).numpy(), ref["Z"], True)


def test_pipelined_rejects_bad_micro_count():
    cfg = S.preset("switch_bf16", T=256, seed=39)
    run = LayerRun(cfg, S.make_inputs(cfg, device="cuda"))
    for bad in (0, C.load() and 65):
        with pytest.raises(C.Ec2moeError):
            C.ec2moe_layer_forward_pipelined(run.desc, run.weights, run.inp["X"], run.mask, run.Y, run.topk_idx,
                                             run.topk_w, run.counts, run.Z, run.workspace, run.ws_bytes, bad)
    assert C.ec2moe_pipelined_workspace_size(run.desc, 0) == 0
