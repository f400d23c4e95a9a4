"""Failure detection without a GPU fault: every wait inside the tensor-core
kernels is bounded.  With a wait budget of 0 the first wait that is not
already satisfied gives up; the CTA drains its own copies and MMAs, frees its
tensor memory and returns, and the host reads EC2MOE_ERR_TIMEOUT.  The same
process then runs the layer normally and gets the same output as before.

Routing reads the caller's Top-k ids on the device, so ids outside [0, E)
cannot be refused before the launch: the routing kernels skip them (no shared
or global access through them) and the host reads EC2MOE_ERR_INVALID_ARG."""
import numpy as np
import pytest
import torch

from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import LayerRun

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()


@pytest.mark.parametrize("cfg", [S.preset("switch_bf16", T=512, seed=31),
                                 S.preset("finegrained_bf16", T=300, seed=32),
                                 # ~2730 rows per expert: the expert GEMMs run on CTA pairs
                                 S.preset("mixtral_bf16", T=4096, E=4, n_allowed=3, d_ff=1024, seed=33),
                                 # two rows: expert GEMMs with the operands swapped, split-K down projection
                                 S.preset("decode_bf16", T=1, d_ff=4096, seed=34)],
                         ids=["switch", "finegrained", "mixtral-pairs", "decode-swap"])
def test_zero_wait_budget_times_out_and_recovers(cfg):
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    y_ref = run.forward().clone()
    assert C.ec2moe_last_device_error() == C.OK
    old = C.ec2moe_get_wait_budget()
    try:
        C.ec2moe_set_wait_budget(0)
        run.forward()
        status = C.ec2moe_last_device_error()
    finally:
        C.ec2moe_set_wait_budget(old)
    assert status == C.ERR_TIMEOUT
    assert C.ec2moe_last_device_error() == C.OK  # the error word was read and cleared
    y = run.forward().clone()
    assert C.ec2moe_last_device_error() == C.OK
    assert torch.equal(y, y_ref)


def test_wait_budget_rejects_negative():
    with pytest.raises(C.Ec2moeError) as e:
        C.ec2moe_set_wait_budget(-1)
    assert e.value.status == C.ERR_INVALID_ARG


@pytest.mark.parametrize("T,k,E", [(300, 2, 16), (9000, 2, 16), (20000, 1, 64)],
                         ids=["one-block", "two-kernel", "two-kernel-E64"])
@pytest.mark.parametrize("noalloc", [False, True], ids=["workspace", "noalloc"])
def test_route_out_of_range_ids_are_skipped_and_reported(T, k, E, noalloc):
    d = 64
    desc = C.make_desc(T=T, d=d, E=E, d_ff=128, k=k)
    g = torch.Generator(device="cuda")
    g.manual_seed(T + E)
    idx = torch.randint(0, E, (T, k), generator=g, device="cuda", dtype=torch.int32)
    bad = [(0, 0), (T // 2, k - 1), (T - 1, 0)]
    for (t, s), v in zip(bad, (E, -1, 1 << 30)):
        idx[t, s] = v
    n = T * k
    X = torch.randn(T, d, generator=g, device="cuda").to(torch.bfloat16)
    counts = torch.empty(E, dtype=torch.int32, device="cuda")
    offsets = torch.empty(E + 1, dtype=torch.int32, device="cuda")
    perm = torch.full((n,), -5, dtype=torch.int32, device="cuda")
    inv = torch.empty(n, dtype=torch.int32, device="cuda")
    dst = torch.zeros(n, d, dtype=torch.bfloat16, device="cuda")
    if noalloc:
        C.ec2moe_route_noalloc(desc, idx, counts, offsets, perm, inv, X, d, dst)
    else:
        wsb = C.ec2moe_route_workspace_size(desc)
        ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
        C.ec2moe_route(desc, idx, counts, offsets, perm, inv, X, d, dst, ws, wsb)
    assert C.ec2moe_last_device_error() == C.ERR_INVALID_ARG
    assert C.ec2moe_last_device_error() == C.OK  # read and cleared
    flat = idx.cpu().numpy().ravel()
    valid = (flat >= 0) & (flat < E)
    assert np.array_equal(counts.cpu().numpy(), np.bincount(flat[valid], minlength=E))
    m = int(valid.sum())
    assert offsets.cpu().numpy()[-1] == m
    p = perm.cpu().numpy()
    assert np.array_equal(np.sort(p[:m]), np.flatnonzero(valid))
    iv = inv.cpu().numpy()
    assert (iv[~valid] == -1).all() and np.array_equal(iv[p[:m]], np.arange(m))
    rows = torch.from_numpy((p[:m] // k).astype(np.int64)).cuda()
    assert torch.equal(dst[:m], X[rows])
    # the context is intact: a valid call afterwards succeeds and reports OK
    idx[idx >= E] = 0
    idx[idx < 0] = 0
    C.ec2moe_route_noalloc(desc, idx, counts, offsets, perm, inv, X, d, dst) if noalloc else \
        C.ec2moe_route(desc, idx, counts, offsets, perm, inv, X, d, dst, ws, wsb)
    assert C.ec2moe_last_device_error() == C.OK
    assert int(counts.sum().item()) == n


# Expert-order tables handed to ec2moe_experts that do not describe the call's
# rows: every grouped GEMM (swapped-operand kernel for <= 16 rows, tensor-core
# kernel, SIMT kernel for fp32) checks each group range against the rows and
# each scatter destination, skips what lies outside, and reports
# EC2MOE_ERR_INVALID_ARG; nothing past the output buffer is written.
EXPERT_SHAPES = [(8, 2, 4, 256, 256, C.BF16), (200, 2, 4, 256, 512, C.BF16), (96, 2, 4, 128, 256, C.F32)]
CORRUPTIONS = ["offset-past-rows", "negative-offset", "decreasing-offsets", "perm-out-of-range"]


@pytest.mark.parametrize("shape", EXPERT_SHAPES, ids=["swapped", "tensor-core", "simt-fp32"])
@pytest.mark.parametrize("bad", CORRUPTIONS)
def test_experts_skip_tables_outside_the_rows(shape, bad):
    T, k, E, d, d_ff, dtype = shape
    n = T * k
    dt = torch.bfloat16 if dtype == C.BF16 else torch.float32
    g = torch.Generator(device="cuda")
    g.manual_seed(77 + T)
    Xp = torch.randn(n, d, generator=g, device="cuda").to(dt)
    W1 = (torch.randn(E, d_ff, d, generator=g, device="cuda") * d ** -0.5).to(dt)
    W3 = (torch.randn(E, d_ff, d, generator=g, device="cuda") * d ** -0.5).to(dt)
    W2 = (torch.randn(E, d, d_ff, generator=g, device="cuda") * d_ff ** -0.5).to(dt)
    rs = np.random.default_rng(T)
    counts = np.bincount(rs.integers(0, E, size=n), minlength=E)
    counts[1] = max(counts[1], 2)
    counts[E - 1] = max(counts[E - 1], 1)
    counts[0] = n - counts[1:].sum()
    assert counts[0] >= 1
    offsets_h = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    perm_h = rs.permutation(n).astype(np.int32)
    w = torch.from_numpy(rs.uniform(0.1, 1.0, size=(T, k)).astype(np.float32)).cuda()
    desc = C.make_desc(T=T, d=d, E=E, d_ff=d_ff, k=k, act=C.SWIGLU, dtype=dtype)
    ews = C.ec2moe_experts_workspace_size(desc)
    ew = torch.empty(max(ews, 16), dtype=torch.uint8, device="cuda")
    guard = 8

    def call(offs, perm):
        slot = torch.full((n + guard, d), 7.0, dtype=dt, device="cuda")
        C.ec2moe_experts(desc, Xp, torch.from_numpy(offs).cuda(), W1, W3, W2, w, torch.from_numpy(perm).cuda(),
                         slot, ew, ews)
        return slot, C.ec2moe_last_device_error()

    ref, status = call(offsets_h, perm_h)
    assert status == C.OK
    assert torch.all(ref[n:] == 7.0)
    offs, perm = offsets_h.copy(), perm_h.copy()
    if bad == "offset-past-rows":
        offs[E] = n + 100
    elif bad == "negative-offset":
        offs[1] = -5
    elif bad == "decreasing-offsets":
        offs[2] = offs[1] - 1
    else:
        perm[3] = n + 1000
    out, status = call(offs, perm)
    assert status == C.ERR_INVALID_ARG
    assert torch.all(out[n:] == 7.0)  # nothing written past the rows
    again, status = call(offsets_h, perm_h)
    assert status == C.OK
    assert torch.equal(again, ref)
