"""Decode-sized expert groups (at most 16 token rows each) against the oracle,
through the expert entry points, on group layouts the layer's routing rarely
produces: one group holding all 16 rows, groups spread over expert ids that
fall in different 32-wide chunks, empty groups, d_ff that is not a multiple of
the 64-column SwiGLU tile and d_model that is not a multiple of the 64-column
K block.  Such groups run on the tensor cores with the operands swapped
(weight rows on the MMA's 128-row side, tokens on its 16-wide side).

EC2MOE_GEMM_SWAP=0 turns that kernel off; a child process then runs these
cases and the decode-sized layer cases on the other kernels (the CUDA-core
weight-streaming GEMM and the usual tensor-core orientation).  The variable is
read once per process."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from oracle import ec2moe_oracle as orc
from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from tests.parity import output_check

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()
    yield
    torch.cuda.synchronize()


def _np(t):
    return t.detach().to("cpu").to(torch.float64).numpy()


def _normal(g, shape, std):
    return (torch.randn(*shape, generator=g, device="cuda", dtype=torch.float32) * std).to(torch.bfloat16)


# (T, k, E, rows per group {expert: rows}, d, d_ff, activation)
ROUTED_CASES = [
    (8, 2, 5, {0: 16}, 288, 224, C.SWIGLU),                    # all 16 rows in one group; ragged N and K
    (8, 2, 100, {0: 3, 37: 1, 64: 7, 99: 5}, 512, 1024, C.SWIGLU),  # groups in four 32-wide id chunks
    (5, 3, 7, {0: 2, 2: 5, 3: 1, 5: 7}, 288, 224, C.GELU),     # empty groups between; ragged shapes
    (1, 1, 3, {1: 1}, 4096, 4096, C.GELU),                     # one row, long K
    (2, 2, 8, {3: 1, 6: 3}, 1024, 2048, C.SWIGLU),
]


@pytest.mark.parametrize("case", ROUTED_CASES, ids=lambda c: f"T{c[0]}-k{c[1]}-E{c[2]}-d{c[4]}-f{c[5]}-act{c[6]}")
def test_routed_experts_small_groups(case):
    T, k, E, rows, d, d_ff, act = case
    n = T * k
    assert sum(rows.values()) == n
    g = torch.Generator(device="cuda")
    g.manual_seed(1000 + E + d)
    counts = np.zeros(E, dtype=np.int64)
    for e, c in rows.items():
        counts[e] = c
    offsets_h = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    Xp = _normal(g, (n, d), 1.0)
    W1 = _normal(g, (E, d_ff, d), d ** -0.5)
    W3 = _normal(g, (E, d_ff, d), d ** -0.5) if act == C.SWIGLU else None
    W2 = _normal(g, (E, d, d_ff), d_ff ** -0.5)
    rs = np.random.default_rng(E * 7 + n)
    perm_h = rs.permutation(n).astype(np.int32)
    w_h = rs.uniform(0.1, 1.0, size=(T, k)).astype(np.float32)
    offsets = torch.from_numpy(offsets_h).cuda()
    perm = torch.from_numpy(perm_h).cuda()
    w = torch.from_numpy(w_h).cuda()
    desc = C.make_desc(T=T, d=d, E=E, d_ff=d_ff, k=k, act=act, dtype=C.BF16)
    ews = C.ec2moe_experts_workspace_size(desc)
    ew = torch.empty(max(ews, 16), dtype=torch.uint8, device="cuda")
    slot = torch.full((n, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    C.ec2moe_experts(desc, Xp, offsets, W1, W3, W2, w, perm, slot, ew, ews)
    torch.cuda.synchronize()
    assert C.ec2moe_last_device_error() == C.OK

    ref = np.zeros((n, d))
    xp = _np(Xp)
    wf = w_h.reshape(-1).astype(np.float64)
    for e in range(E):
        lo, hi = int(offsets_h[e]), int(offsets_h[e + 1])
        if hi == lo:
            continue
        y = orc.expert_ffn(xp[lo:hi], _np(W1[e]), _np(W2[e]), None if W3 is None else _np(W3[e]), act)
        for p in range(lo, hi):
            ref[perm_h[p]] = wf[perm_h[p]] * y[p - lo]
    out = _np(slot)
    assert np.isfinite(out).all()  # every slot written
    output_check(out, ref, True)


@pytest.mark.parametrize("T,n_shared,d,fs,act", [(5, 2, 288, 224, C.SWIGLU), (16, 1, 512, 1024, C.GELU),
                                                 (1, 3, 1024, 512, C.SWIGLU)])
def test_shared_experts_small_batches(T, n_shared, d, fs, act):
    g = torch.Generator(device="cuda")
    g.manual_seed(2000 + T + d)
    Xh = _normal(g, (T, d), 1.0)
    W1s = _normal(g, (n_shared, fs, d), d ** -0.5)
    W3s = _normal(g, (n_shared, fs, d), d ** -0.5) if act == C.SWIGLU else None
    W2s = _normal(g, (n_shared, d, fs), fs ** -0.5)
    desc = C.make_desc(T=T, d=d, E=4, d_ff=256, k=1, act=act, dtype=C.BF16, n_shared=n_shared, d_ff_shared=fs)
    ews = C.ec2moe_experts_workspace_size(desc)
    ew = torch.empty(max(ews, 16), dtype=torch.uint8, device="cuda")
    shared = torch.full((n_shared * T, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    C.ec2moe_shared_experts(desc, Xh, W1s, W3s, W2s, shared, ew, ews)
    torch.cuda.synchronize()
    assert C.ec2moe_last_device_error() == C.OK
    xh = _np(Xh)
    ref = np.concatenate([orc.expert_ffn(xh, _np(W1s[j]), _np(W2s[j]), None if W3s is None else _np(W3s[j]), act)
                          for j in range(n_shared)])
    out = _np(shared)
    assert np.isfinite(out).all()
    output_check(out, ref, True)


LAYER_SELECT = "test_layer_forward and (decode_bf16 or T2- or T3-)"


def test_small_groups_with_swap_kernel_off():
    if os.environ.get("EC2MOE_GEMM_SWAP") == "0":
        pytest.skip("already the child process")
    env = dict(os.environ, EC2MOE_GEMM_SWAP="0")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_gpu_parity.py"),
                        os.path.join(ROOT, "tests", "test_gpu_swap.py"), "-k",
                        f"({LAYER_SELECT}) or test_routed_experts_small_groups or test_shared_experts_small_batches"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
