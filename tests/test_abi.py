"""The C-ABI library loads and exports every symbol include/ec2moe.h declares, and
its host-side checks reject bad arguments before touching the GPU (CPU only:
only calls that fail validation, or that have nothing to do, are made)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ec2moe.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return C.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ec2moe_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ["ec2moe_gate", "ec2moe_route", "ec2moe_experts", "ec2moe_combine", "ec2moe_lr_encode",
              "ec2moe_lr_decode", "ec2moe_layer_forward"]:
        assert n in names
    assert set(names) == set(C.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    for n in declared_functions():
        assert hasattr(lib, n), n


def _desc(**kw):
    base = dict(T=64, d=256, E=8, d_ff=512, k=2, n_groups=2, act=C.GELU, dtype=C.BF16, r=64)
    base.update(kw)
    return C.make_desc(**base)


BAD = 0x1001  # never dereferenced: validation fails first


def _status(fn, *args):
    try:
        fn(*args)
    except C.Ec2moeError as e:
        return e.status
    return C.OK


def test_gate_rejections(lib):
    ok_mask = np.ones(8, np.uint8)
    A = 0x100000  # aligned fake address, never reached
    g = lambda desc, mask, X=A: _status(C.ec2moe_gate, desc, X, A, A, A, A, mask, A, A, 0)
    assert g(_desc(), np.zeros(8, np.uint8)) == C.ERR_ALL_MASKED
    assert g(_desc(k=3), np.array([1, 1, 0, 0, 0, 0, 0, 0], np.uint8)) == C.ERR_TOO_FEW_EXPERTS
    assert g(_desc(E=9), np.ones(9, np.uint8)) == C.ERR_INVALID_ARG  # E % K != 0
    assert g(_desc(E=256, n_groups=1), np.ones(256, np.uint8)) == C.ERR_UNSUPPORTED
    assert g(_desc(k=9), ok_mask) == C.ERR_TOO_FEW_EXPERTS
    assert g(_desc(d=260), ok_mask) == C.ERR_MISALIGNED
    assert g(_desc(), ok_mask, X=BAD) == C.ERR_MISALIGNED
    assert g(_desc(), ok_mask, X=0) == C.ERR_INVALID_ARG
    assert g(_desc(act=7), ok_mask) == C.ERR_INVALID_ARG
    assert g(_desc(dtype=5), ok_mask) == C.ERR_INVALID_ARG
    assert g(_desc(T=-1), ok_mask) == C.ERR_INVALID_ARG
    assert g(_desc(T=0), ok_mask) == C.OK  # nothing to do, nothing launched
    assert C.ec2moe_last_launch_count() == 0
    assert _status(C.ec2moe_gate, None, A, A, A, A, A, ok_mask, A, A, 0) == C.ERR_INVALID_ARG


def test_layer_rejections(lib):
    A = 0x100000
    w = C.make_weights(W_local=A, b_local=A, W_global=A, b_global=A, W1=A, W2=A, V_enc=A, V_dec=A)
    mask = np.ones(8, np.uint8)
    f = lambda desc, ws=A, wsb=1 << 40, mask=mask, w=w: _status(
        C.ec2moe_layer_forward, desc, w, A, mask, A, A, A, A, None, ws, wsb, 0)
    d = _desc()
    assert f(d, ws=A, wsb=C.ec2moe_workspace_size(d) - 1) == C.ERR_WORKSPACE
    assert f(d, ws=None) == C.ERR_WORKSPACE
    assert f(d, ws=BAD) == C.ERR_MISALIGNED
    assert f(_desc(d_ff=520)) == C.ERR_UNSUPPORTED  # tensor-core tiles need multiples of 32
    assert f(_desc(r=36)) == C.ERR_MISALIGNED
    assert f(_desc(act=C.SWIGLU)) == C.ERR_INVALID_ARG  # W3 missing
    assert f(_desc(), mask=np.zeros(8, np.uint8)) == C.ERR_ALL_MASKED
    w2 = C.make_weights(W_local=A, b_local=A, W1=A, W2=A, V_enc=A, V_dec=A)
    assert f(_desc(), w=w2) == C.ERR_INVALID_ARG  # K = 2 needs the global gate
    assert f(_desc(T=0)) == C.OK


def test_workspace_sizes(lib):
    d = _desc(T=1000, k=2, E=8, d=256, d_ff=512, r=64)
    ws = C.ec2moe_workspace_size(d)
    es = 2
    need = (1000 * 64 * es) + (3000 * 256 * es) + (2000 * 512 * es) + (2000 * 256 * es) + 2 * 2000 * 4
    assert ws >= need and ws < need + 64 * 1024
    assert C.ec2moe_experts_workspace_size(d) >= 2000 * 512 * es
    assert C.ec2moe_route_workspace_size(d) >= 2 * 8 * 4
    assert C.ec2moe_workspace_size(_desc(E=9)) == 0


def test_workspace_covers_decode_regions(lib):
    """Decode-sized bf16 calls add fp32 partial-sum regions: the small-batch
    gate's [d/128, T, E+K] logits, the split-K encoder's [<=32, T, r] and the
    split-K down projection's [<=8, T*k, d]; larger batches add none of them."""
    T, d, E, K, k, r, ff = 64, 4096, 8, 2, 2, 256, 14336
    ws = C.ec2moe_workspace_size(_desc(T=T, d=d, E=E, n_groups=K, k=k, r=r, d_ff=ff))
    es = 2
    dense = (T * r + (T * k + T) * d + T * k * ff + T * k * d) * es
    partials = (d // 128) * T * (E + K) * 4 + 32 * T * r * 4 + 8 * T * k * d * 4
    assert ws >= dense + partials
    big = C.ec2moe_workspace_size(_desc(T=300, d=d, E=E, n_groups=K, k=k, r=r, d_ff=ff))
    big_dense = (300 * r + (300 * k + 300) * d + 300 * k * ff + 300 * k * d) * es
    assert big_dense <= big < big_dense + 4 * 1024 * 1024  # no T-sized partial regions


def test_other_entry_points_validate(lib):
    A = 0x100000
    d = _desc()
    assert _status(C.ec2moe_route, d, A, A, A, A, None, None, 0, None, None, 0, 0) == C.ERR_WORKSPACE
    assert _status(C.ec2moe_route, d, A, A, A, A, None, A, 0, A, A, 1 << 20, 0) == C.ERR_INVALID_ARG
    assert _status(C.ec2moe_experts, d, A, A, A, None, A, A, A, A, None, 0, 0) == C.ERR_WORKSPACE
    assert _status(C.ec2moe_experts, _desc(act=C.SWIGLU), A, A, A, None, A, A, A, A, A, 1 << 30, 0) == C.ERR_INVALID_ARG
    assert _status(C.ec2moe_lr_encode, _desc(r=0), A, A, A, 0) == C.ERR_INVALID_ARG
    assert _status(C.ec2moe_lr_decode, d, A, BAD, A, 0) == C.ERR_MISALIGNED
    assert _status(C.ec2moe_combine, d, BAD, None, A, 0) == C.ERR_MISALIGNED
    assert _status(C.ec2moe_shared_experts, _desc(n_shared=1, d_ff_shared=0), A, A, None, A, A, A, 1 << 30, 0) == \
        C.ERR_INVALID_ARG
    assert C.status_string(C.ERR_TIMEOUT) == "device wait timed out"


def test_top_group_pruning_validation(lib):
    """Top-group pruning is checked on the host: a negative count is invalid,
    and k above the allowed experts of the fewest-member choice of kept groups
    is refused (the same rule as the oracle's pruned_candidate_floor)."""
    from oracle import ec2moe_oracle as orc
    A = 0x100000
    mask = np.array([1, 0, 0, 0, 1, 1, 1, 0], np.uint8)  # groups of 2: allowed counts 1, 0, 2, 1
    for G, k in [(1, 1), (1, 2), (2, 2), (2, 3), (3, 4), (3, 3), (0, 4)]:
        d = _desc(T=0, E=8, n_groups=4, k=k, top_groups=G)  # T = 0: validation only, nothing to launch
        got = _status(C.ec2moe_gate, d, A, A, A, A, A, mask, A, A, 0)
        floor_k = orc.pruned_candidate_floor(mask.astype(bool), 4, G) if G else int(mask.sum())
        want = C.ERR_TOO_FEW_EXPERTS if k > floor_k else C.OK
        assert got == want, (G, k, got)
    assert _status(C.ec2moe_gate, _desc(n_groups=2, top_groups=-1), A, A, A, A, A, np.ones(8, np.uint8), A, A, 0) == \
        C.ERR_INVALID_ARG
    assert _status(C.ec2moe_profile_only, -2) == C.ERR_INVALID_ARG
