"""ec2moe_route_noalloc: routing for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc: a serving process that reserves all device
memory for its own pool before it starts, a latency-critical loop that must not
pay cudaMalloc's implicit device synchronisation, or a foreign-language binding
without a device allocator.  For them the library keeps the routing histograms
in a fixed device array of its own.  These tests check that the scratch-free
entry point returns exactly what ec2moe_route (caller workspace) returns, on
two calls in a row (the shared array keeps the first call's contents), and that
sizes beyond the array are refused before anything runs.  This file is
collected last on purpose.
"""
import numpy as np
import pytest
import torch

from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import desc_for


@pytest.fixture(scope="module")
def lib():
    B.build()
    return C.load()


def test_oversize_is_refused_before_any_launch(lib):
    # ceil(T*k/1024) * E cells must fit EC2MOE_ROUTE_NOALLOC_MAX_CELLS = 16384
    A = 0x100000  # aligned placeholder address, never dereferenced
    big = C.make_desc(T=262145, d=256, E=64, d_ff=512, k=1)
    with pytest.raises(C.Ec2moeError) as e:
        C.ec2moe_route_noalloc(big, A, A, A, A, None, None, 0, None, 0)
    assert e.value.status == C.ERR_UNSUPPORTED
    assert C.ec2moe_last_launch_count() == 0


def _route_both(cfg, X):
    """Routes one batch with both entry points; returns both result sets."""
    desc = desc_for(cfg)
    inp = S.make_inputs(cfg, device="cuda", with_experts=False)
    idx = torch.empty((cfg.T, cfg.k), dtype=torch.int32, device="cuda")
    w = torch.empty((cfg.T, cfg.k), dtype=torch.float32, device="cuda")
    C.ec2moe_gate(desc, inp["X"], inp["W_local"], inp["b_local"], inp["W_global"], inp["b_global"],
                  inp["mask"].cpu(), idx, w)
    n = cfg.T * cfg.k
    outs = []
    for use_noalloc in (False, True):
        counts = torch.full((cfg.E,), -7, dtype=torch.int32, device="cuda")
        offsets = torch.full((cfg.E + 1,), -7, dtype=torch.int32, device="cuda")
        perm = torch.full((n,), -7, dtype=torch.int32, device="cuda")
        inv = torch.full((n,), -7, dtype=torch.int32, device="cuda")
        dst = torch.zeros((n, cfg.d), dtype=X.dtype, device="cuda")
        if use_noalloc:
            C.ec2moe_route_noalloc(desc, idx, counts, offsets, perm, inv, X, cfg.d, dst)
        else:
            wsb = C.ec2moe_route_workspace_size(desc)
            ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
            C.ec2moe_route(desc, idx, counts, offsets, perm, inv, X, cfg.d, dst, ws, wsb)
        outs.append((counts, offsets, perm, inv, dst))
    torch.cuda.synchronize()
    return idx, outs


@pytest.mark.gpu
def test_noalloc_route_matches_workspace_route_twice(lib):
    # Two calls in a row, both with more than 16384 (token, slot) entries so
    # that both take the two-kernel routing that reads the library's array,
    # and with different expert counts (64, then 16): the second call's kernels
    # run over cells the first call left behind in another layout.
    for cfg in (S.preset("finegrained_bf16", T=9000, seed=21),
                S.preset("switch_bf16", T=20000, k=2, n_groups=4, seed=22)):
        assert cfg.T * cfg.k > 16384
        X = S.make_inputs(cfg, device="cuda", with_experts=False)["X"]
        idx, (ref, got) = _route_both(cfg, X)
        for a, b in zip(ref, got):
            assert torch.equal(a, b)
        counts = got[0].cpu().numpy()
        assert np.array_equal(counts, np.bincount(idx.cpu().numpy().ravel(), minlength=cfg.E))
    assert C.ec2moe_last_device_error() == C.OK


@pytest.mark.gpu
def test_noalloc_route_at_the_array_limit(lib):
    # ceil(T*k/1024) * E = 256 * 64 = 16384 cells: exactly the array's size.
    T, E, k = 262144, 64, 1
    desc = C.make_desc(T=T, d=256, E=E, d_ff=512, k=k)
    g = torch.Generator(device="cuda")
    g.manual_seed(31)
    outs = []
    for seed_shift in (0, 1):
        idx = torch.randint(0, E, (T, k), generator=g, device="cuda", dtype=torch.int32)
        res = []
        for use_noalloc in (False, True):
            counts = torch.full((E,), -7, dtype=torch.int32, device="cuda")
            offsets = torch.full((E + 1,), -7, dtype=torch.int32, device="cuda")
            perm = torch.full((T * k,), -7, dtype=torch.int32, device="cuda")
            if use_noalloc:
                C.ec2moe_route_noalloc(desc, idx, counts, offsets, perm)
            else:
                wsb = C.ec2moe_route_workspace_size(desc)
                ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
                C.ec2moe_route(desc, idx, counts, offsets, perm, None, None, 0, None, ws, wsb)
            res.append((counts, offsets, perm))
        torch.cuda.synchronize()
        for a, b in zip(*res):
            assert torch.equal(a, b)
        assert np.array_equal(res[1][0].cpu().numpy(), np.bincount(idx.cpu().numpy().ravel(), minlength=E))
        outs.append(res[1][2].clone())
    assert not torch.equal(outs[0], outs[1])
    assert C.ec2moe_last_device_error() == C.OK
