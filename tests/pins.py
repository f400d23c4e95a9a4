"""Pins for the fp64 oracle: checks against facts fixed by the paper's definitions
and by mathematics, never against the oracle itself.

Each ``pin_*`` takes the oracle module and raises AssertionError (or the
oracle's own ValueError) when it disagrees.  ``test_oracle_pins`` runs them on
the oracle; ``test_oracle_mutants`` plants plausible mistakes in the oracle and
checks that some pin catches each one.
"""

from __future__ import annotations

import itertools
import json
import math
import os

import numpy as np
from scipy.special import expit, softmax
from scipy.stats import norm

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "worked_examples.json")


def _num(v):
    if isinstance(v, str):
        return {"ln2": math.log(2.0), "ln3": math.log(3.0), "ln4": math.log(4.0), "ln5": math.log(5.0),
                "ln3-0.5": math.log(3.0) - 0.5, "ln3-ln2": math.log(1.5)}[v]
    return float(v)


def golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _gate_example():
    ex = golden()["group_gate"]
    x = np.array(ex["x"])[None, :]
    Wl = np.array([[_num(v) for v in row] for row in ex["W_local"]])
    bl = np.array([_num(v) for v in ex["b_local"]])
    Wg = np.array([[_num(v) for v in row] for row in ex["W_global"]])
    bg = np.array([_num(v) for v in ex["b_global"]])
    return ex, x, Wl, bl, Wg, bg


def _rand_gate(rng, T, d, E, K):
    X = rng.standard_normal((T, d))
    Wl = rng.standard_normal((E, d)) / math.sqrt(d)
    bl = 0.3 * rng.standard_normal(E)
    Wg = rng.standard_normal((K, d)) / math.sqrt(d) if K > 1 else None
    bg = 0.3 * rng.standard_normal(K) if K > 1 else None
    return X, Wl, bl, Wg, bg


# ---------------------------------------------------------------- gate (Eq. 4-7)

def pin_gate_golden(orc):
    """Hand-derived g and top-k of the worked example (closed forms)."""
    ex, x, Wl, bl, Wg, bg = _gate_example()
    for case in ex["cases"]:
        mask = np.array(case["mask"], dtype=np.uint8)
        r = orc.gate_and_route(x, Wl, bl, Wg, bg, mask, ex["n_groups"], 1)
        np.testing.assert_allclose(r["g"][0], case["g"], rtol=0, atol=1e-12)
        assert r["idx"][0].tolist() == case["top1"]
        r2 = orc.gate_and_route(x, Wl, bl, Wg, bg, mask, ex["n_groups"], 2)
        assert r2["idx"][0].tolist() == case["top2"]
        if case["top3"] is None:
            try:
                orc.gate_and_route(x, Wl, bl, Wg, bg, mask, ex["n_groups"], 3)
            except ValueError:
                pass
            else:
                raise AssertionError("k above the allowed count must be rejected")
        else:
            r3 = orc.gate_and_route(x, Wl, bl, Wg, bg, mask, ex["n_groups"], 3)
            assert r3["idx"][0].tolist() == case["top3"]
    # decision margins in log g: top-1 of the unmasked case sits on a tie (gap 0);
    # top-2 clears expert 1 by ln((3/8)/(3/16)) = ln 2 with a tie inside the top-2.
    r2 = orc.gate_and_route(x, Wl, bl, Wg, bg, np.ones(4, np.uint8), ex["n_groups"], 2)
    np.testing.assert_allclose(r2["gap_boundary"], [math.log(2.0)], atol=1e-12)
    np.testing.assert_allclose(r2["gap_adjacent"], [[0.0]], atol=1e-12)
    r1 = orc.gate_and_route(x, Wl, bl, Wg, bg, np.ones(4, np.uint8), ex["n_groups"], 1)
    np.testing.assert_allclose(r1["gap_boundary"], [0.0], atol=1e-12)
    sg = ex["single_group"]
    r = orc.gate_and_route(x, Wl, bl, None, None, np.array(sg["mask"], np.uint8), 1, 2)
    np.testing.assert_allclose(r["g"][0], sg["g"], rtol=0, atol=1e-12)
    assert r["idx"][0].tolist() == sg["top2"]


def pin_gate_sums_to_one(orc, seed=1):
    """Eq. 1 requires sum_i G(x)_i = 1; Eq. 5-7 give it over the allowed experts."""
    rng = np.random.default_rng(seed)
    for (E, K) in [(8, 2), (16, 1), (64, 8), (12, 3)]:
        X, Wl, bl, Wg, bg = _rand_gate(rng, 40, 24, E, K)
        for _ in range(4):
            mask = (rng.random(E) < 0.5).astype(np.uint8)
            mask[rng.integers(E)] = 1
            l, m = orc.gate_logits(X, Wl, bl, Wg, bg)
            g, log_g = orc.group_gate(l, m, mask.astype(bool), K)
            np.testing.assert_allclose(g.sum(axis=1), 1.0, rtol=0, atol=1e-12)
            assert np.all(g[:, mask == 0] == 0.0)
            assert np.all(g[:, mask == 1] > 0.0)
            np.testing.assert_allclose(np.exp(log_g[:, mask == 1]), g[:, mask == 1], rtol=1e-12, atol=0)


def pin_masked_never_selected(orc, seed=2):
    """Eq. 4: experts outside the local set are never candidates, even with huge logits."""
    rng = np.random.default_rng(seed)
    E, K, k = 16, 4, 3
    X, Wl, bl, Wg, bg = _rand_gate(rng, 64, 16, E, K)
    mask = np.ones(E, np.uint8)
    mask[[1, 5, 6, 7, 12]] = 0
    bl = bl.copy()
    bl[[1, 5, 6, 7, 12]] = 50.0  # masked experts would win every token
    r = orc.gate_and_route(X, Wl, bl, Wg, bg, mask, K, k)
    assert not np.isin(r["idx"], [1, 5, 6, 7, 12]).any()


def pin_single_group_is_softmax(orc, seed=3):
    """K = 1 reduces the two-stage gate to one masked softmax (scipy.special.softmax)."""
    rng = np.random.default_rng(seed)
    E = 10
    X, Wl, bl, _, _ = _rand_gate(rng, 30, 12, E, 1)
    mask = np.array([1, 0, 1, 1, 0, 1, 1, 1, 0, 1], np.uint8)
    r = orc.gate_and_route(X, Wl, bl, None, None, mask, 1, 2)
    logits = X @ Wl.T + bl
    ref = softmax(logits[:, mask == 1], axis=1)
    np.testing.assert_allclose(r["g"][:, mask == 1], ref, rtol=1e-12, atol=1e-15)


def pin_group_factorisation(orc, seed=4):
    """Eq. 7 factorises: summing g over a group gives that group's p_group, which is
    scipy's softmax of the global logits over live groups; within a group, g is
    proportional to scipy's softmax of the local logits."""
    rng = np.random.default_rng(seed)
    E, K = 12, 3
    X, Wl, bl, Wg, bg = _rand_gate(rng, 25, 10, E, K)
    mask = np.ones(E, np.uint8)
    mask[[0, 1, 2, 3]] = 0  # group 0 dead
    mask[[5, 9]] = 0
    l, m = orc.gate_logits(X, Wl, bl, Wg, bg)
    g, _ = orc.group_gate(l, m, mask.astype(bool), K)
    pg = softmax((X @ Wg.T + bg)[:, 1:], axis=1)
    np.testing.assert_allclose(g[:, 4:8].sum(1), pg[:, 0], rtol=1e-12)
    np.testing.assert_allclose(g[:, 8:12].sum(1), pg[:, 1], rtol=1e-12)
    loc = softmax((X @ Wl.T + bl)[:, [4, 6, 7]], axis=1)
    np.testing.assert_allclose(g[:, [4, 6, 7]] / pg[:, :1], loc, rtol=1e-12)


def pin_topk_bruteforce(orc, seed=5):
    """Top-k equals exhaustive enumeration of k-subsets (max sum of g; among equal
    sums the lexicographically smallest index tuple), with slots ordered by
    (g descending, index ascending).  Logits on a coarse grid force many ties."""
    rng = np.random.default_rng(seed)
    E = 8
    for K, k in [(1, 1), (2, 2), (4, 3), (1, 4)]:
        T = 48
        X = rng.integers(-2, 3, size=(T, 4)).astype(np.float64)
        Wl = rng.integers(-1, 2, size=(E, 4)).astype(np.float64) * 0.5
        bl = np.zeros(E)
        Wg = rng.integers(-1, 2, size=(K, 4)).astype(np.float64) * 0.5 if K > 1 else None
        bg = np.zeros(K) if K > 1 else None
        mask = np.ones(E, np.uint8)
        mask[rng.choice(E, 2, replace=False)] = 0
        r = orc.gate_and_route(X, Wl, bl, Wg, bg, mask, K, k)
        g = r["g"]
        allowed = np.nonzero(mask)[0].tolist()
        for t in range(T):
            best, best_key = None, None
            for sub in itertools.combinations(allowed, k):
                s = float(np.sum(g[t, list(sub)]))
                key = (-round(s, 12), sub)
                if best_key is None or key < best_key:
                    best_key, best = key, sub
            got = r["idx"][t].tolist()
            assert sorted(got) == list(best), (t, got, best)
            for a, b in zip(got[:-1], got[1:]):
                assert (g[t, a] > g[t, b]) or (g[t, a] == g[t, b] and a < b)


def pin_rejections(orc):
    """An empty local set, or fewer allowed experts than k, is an error."""
    for mask, k in [(np.zeros(4, np.uint8), 1), (np.array([1, 0, 0, 0], np.uint8), 2)]:
        try:
            orc.allowed_experts(mask, k)
        except ValueError:
            continue
        raise AssertionError("mask must be rejected")


# ------------------------------------------------------------- routing tables

def pin_route_golden(orc):
    ex = golden()["route_tables"]
    for sfx in ["", "_top2"]:
        c, o, p = orc.route_tables(np.array(ex["idx" + sfx]), ex["E"])
        assert c.tolist() == ex["counts" + sfx]
        assert o.tolist() == ex["offsets" + sfx]
        assert p.tolist() == ex["perm" + sfx]


def pin_route_invariants(orc, seed=6):
    """counts sum to T*k and equal a bincount; perm is a bijection that groups rows
    by expert in increasing (token, slot) order."""
    rng = np.random.default_rng(seed)
    T, k, E = 300, 3, 11
    idx = np.stack([rng.choice(E, k, replace=False) for _ in range(T)])
    c, o, p = orc.route_tables(idx, E)
    assert c.sum() == T * k
    assert np.array_equal(c, np.bincount(idx.ravel(), minlength=E))
    assert o[0] == 0 and o[-1] == T * k and np.all(np.diff(o) == c)
    assert np.array_equal(np.sort(p), np.arange(T * k))
    flat = idx.ravel()
    for e in range(E):
        rows = p[o[e]:o[e + 1]]
        assert np.all(flat[rows] == e)
        assert np.all(np.diff(rows) > 0)


# ------------------------------------------------------------------- codec

def pin_codec_golden(orc):
    ex = golden()["codec"]
    Z = orc.lr_encode(np.array(ex["X"]), np.array(ex["V_enc"]))
    np.testing.assert_allclose(Z, ex["Z"], atol=1e-12)
    Xh = orc.lr_decode(Z, np.array(ex["V_dec"]))
    np.testing.assert_allclose(Xh, ex["X_hat"], atol=1e-12)


def pin_codec_identity(orc, seed=7):
    """r = d with orthogonal V_enc = Q^T, V_dec = Q reconstructs X exactly."""
    rng = np.random.default_rng(seed)
    d = 24
    Q, _ = np.linalg.qr(rng.standard_normal((d, d)))
    X = rng.standard_normal((17, d))
    Xh = orc.lr_decode(orc.lr_encode(X, Q.T), Q)
    np.testing.assert_allclose(Xh, X, rtol=0, atol=1e-12)


def pin_codec_projection(orc, seed=8):
    """r < d with orthonormal columns: decode(encode(.)) is the orthogonal projection
    onto span(Q_r): idempotent, and the residual is orthogonal to the span."""
    rng = np.random.default_rng(seed)
    d, r = 20, 6
    Q, _ = np.linalg.qr(rng.standard_normal((d, d)))
    Qr = Q[:, :r]
    X = rng.standard_normal((9, d))
    P = orc.lr_decode(orc.lr_encode(X, Qr.T), Qr)
    P2 = orc.lr_decode(orc.lr_encode(P, Qr.T), Qr)
    np.testing.assert_allclose(P2, P, atol=1e-12)
    np.testing.assert_allclose((X - P) @ Qr, 0.0, atol=1e-12)
    assert orc.lr_encode(X, Qr.T).shape == (9, r)


# ---------------------------------------------------------------- experts

def pin_ffn_golden(orc):
    ex = golden()["expert_ffn"]
    x = np.array(ex["x"])[None, :]
    o = orc.expert_ffn(x, np.array(ex["W1"]), np.array(ex["W2"]), None, orc.GELU)
    np.testing.assert_allclose(o[0], ex["gelu_out"], rtol=0, atol=1e-12)
    o = orc.expert_ffn(x, np.array(ex["W1"]), np.array(ex["W2"]), np.array(ex["W3"]), orc.SWIGLU)
    np.testing.assert_allclose(o[0], ex["swiglu_out"], rtol=0, atol=1e-12)


def pin_activations_library(orc):
    """GELU(u) = u * Phi(u) (scipy.stats.norm.cdf); SiLU(u) = u * sigmoid(u) (scipy.special.expit)."""
    u = np.linspace(-8, 8, 161)
    np.testing.assert_allclose(orc.gelu(u), u * norm.cdf(u), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(orc.silu(u), u * expit(u), rtol=1e-13, atol=1e-15)


def pin_ffn_bruteforce(orc, seed=9):
    """Scalar triple loops on a tiny non-square expert (catches transposed operands)."""
    rng = np.random.default_rng(seed)
    n, d, f = 3, 5, 4
    x = rng.standard_normal((n, d))
    W1, W3 = rng.standard_normal((f, d)), rng.standard_normal((f, d))
    W2 = rng.standard_normal((d, f))
    for act in (orc.GELU, orc.SWIGLU):
        got = orc.expert_ffn(x, W1, W2, W3, act)
        for i in range(n):
            h = []
            for j in range(f):
                a = sum(W1[j, c] * x[i, c] for c in range(d))
                if act == orc.GELU:
                    h.append(a * norm.cdf(a))
                else:
                    b = sum(W3[j, c] * x[i, c] for c in range(d))
                    h.append(a * expit(a) * b)
            for c in range(d):
                ref = sum(W2[c, j] * h[j] for j in range(f))
                assert abs(got[i, c] - ref) <= 1e-12 * (1 + abs(ref)), (act, i, c)


# ------------------------------------------------------------------ layer

def _rand_layer(rng, T, d, E, f, K, act, r, n_shared=0, same_experts=False):
    X, Wl, bl, Wg, bg = _rand_gate(rng, T, d, E, K)
    shp = (1 if same_experts else E, f, d)
    W1 = rng.standard_normal(shp) / math.sqrt(d)
    W3 = rng.standard_normal(shp) / math.sqrt(d)
    W2 = rng.standard_normal((shp[0], d, f)) / math.sqrt(f)
    if same_experts:
        W1, W3, W2 = (np.repeat(a, E, axis=0) for a in (W1, W3, W2))
    inp = dict(X=X, W_local=Wl, b_local=bl, W_global=Wg, b_global=bg, W1=W1,
               W3=W3 if act == 1 else None, W2=W2, W1s=None, W3s=None, W2s=None,
               V_enc=None, V_dec=None)
    if n_shared:
        inp["W1s"], inp["W3s"], inp["W2s"] = W1[:n_shared].copy(), (W3[:n_shared].copy() if act == 1 else None), W2[:n_shared].copy()
    if r:
        inp["V_enc"] = rng.standard_normal((r, d)) / math.sqrt(d)
        inp["V_dec"] = rng.standard_normal((d, r)) / math.sqrt(r)
    return inp


def pin_layer_single_expert(orc, seed=10):
    """E = 1, k = 1, K = 1: g = 1 and the layer is one dense FFN (brute-force loops)."""
    rng = np.random.default_rng(seed)
    for act in (orc.GELU, orc.SWIGLU):
        inp = _rand_layer(rng, 4, 6, 1, 5, 1, act, 0)
        inp["mask"] = np.ones(1, np.uint8)
        out = orc.layer_forward(inp, 1, 1, act)
        np.testing.assert_allclose(out["w"], 1.0, atol=1e-15)
        X, W1, W2, W3 = inp["X"], inp["W1"][0], inp["W2"][0], inp["W3"]
        for i in range(4):
            h = []
            for j in range(5):
                a = sum(W1[j, c] * X[i, c] for c in range(6))
                if act == orc.GELU:
                    h.append(a * norm.cdf(a))
                else:
                    b = sum(W3[0][j, c] * X[i, c] for c in range(6))
                    h.append(a * expit(a) * b)
            for c in range(6):
                ref = sum(W2[c, j] * h[j] for j in range(5))
                assert abs(out["y"][i, c] - ref) <= 1e-12 * (1 + abs(ref))


def pin_layer_linearity(orc, seed=11):
    """With every expert identical, y = (sum of top-k weights + n_shared) * FFN(x_hat);
    with renormalised top-k weights the routed part is exactly FFN(x_hat)."""
    rng = np.random.default_rng(seed)
    for act, K, k, r, ns in [(orc.GELU, 2, 2, 0, 0), (orc.SWIGLU, 4, 3, 6, 2), (orc.GELU, 1, 1, 5, 1)]:
        E, d, f = 8, 10, 7
        inp = _rand_layer(rng, 12, d, E, f, K, act, r, n_shared=ns, same_experts=True)
        inp["mask"] = np.array([1, 1, 0, 1, 1, 1, 0, 1], np.uint8)
        Xh = inp["X"] if r == 0 else (inp["X"] @ inp["V_enc"].T) @ inp["V_dec"].T
        ffn = orc.expert_ffn(Xh, inp["W1"][0], inp["W2"][0], None if inp["W3"] is None else inp["W3"][0], act)
        for renorm in (False, True):
            out = orc.layer_forward(inp, K, k, act, renorm=renorm)
            scale = out["w"].sum(axis=1) + ns
            if renorm:
                np.testing.assert_allclose(out["w"].sum(axis=1), 1.0, atol=1e-12)
            np.testing.assert_allclose(out["y"], scale[:, None] * ffn, rtol=1e-11, atol=1e-12)


def pin_layer_codec_golden(orc):
    """The experts consume the decoded activations: on the worked codec example the
    second token decodes to 0, so a bias-free FFN returns exactly 0 for it."""
    ex = golden()["codec"]
    X = np.array(ex["X"])
    f = 3
    rng = np.random.default_rng(12)
    inp = dict(X=X, W_local=np.zeros((2, 2)), b_local=np.array([0.0, 1.0]), W_global=None, b_global=None,
               mask=np.array([1, 1], np.uint8), W1=rng.standard_normal((2, f, 2)), W3=None,
               W2=rng.standard_normal((2, 2, f)), W1s=None, W3s=None, W2s=None,
               V_enc=np.array(ex["V_enc"]), V_dec=np.array(ex["V_dec"]))
    out = orc.layer_forward(inp, 1, 1, orc.GELU)
    np.testing.assert_allclose(out["Z"], ex["Z"], atol=1e-12)
    np.testing.assert_allclose(out["y"][1], 0.0, atol=1e-15)
    assert np.abs(out["y"][0]).max() > 1e-3
    # both tokens prefer expert 1 (bias 1 vs 0, zero gate weights): g = e/(1+e)
    np.testing.assert_allclose(out["w"][:, 0], math.e / (1 + math.e), rtol=1e-13)
    assert out["idx"][:, 0].tolist() == [1, 1]


def pin_layer_pairing_golden(orc):
    """Eq. 1 pairs G(x)_i with E_i(x): three distinct experts, Top-2 with unequal
    weights, two tokens routed to different expert pairs, and the hand-derived
    y of each (GELU, GELU with renormalised weights, SwiGLU).  A routed row that
    met another expert's weights, or a slot scaled by another slot's weight,
    changes y here."""
    ex = golden()["layer_pairing"]
    X = np.array(ex["x"])
    W1, W3, W2 = (np.array(ex[key]) for key in ("W1", "W3", "W2"))
    base = dict(X=X, W_local=np.array([[_num(v) for v in row] for row in ex["W_local"]]),
                b_local=np.array(ex["b_local"]), W_global=None, b_global=None,
                mask=np.array(ex["mask"], np.uint8), W1=W1, W3=None, W2=W2, W1s=None, W3s=None, W2s=None,
                V_enc=None, V_dec=None)
    for act, renorm, key in [(orc.GELU, False, "y_gelu"), (orc.GELU, True, "y_gelu_renorm"),
                             (orc.SWIGLU, False, "y_swiglu")]:
        inp = dict(base, W3=W3 if act == orc.SWIGLU else None)
        out = orc.layer_forward(inp, ex["n_groups"], ex["k"], act, renorm=renorm)
        assert out["idx"].tolist() == ex["idx"]
        w = np.array(ex["w"])
        if renorm:
            w = w / w.sum(axis=1, keepdims=True)
        np.testing.assert_allclose(out["w"], w, rtol=0, atol=1e-15)
        np.testing.assert_allclose(out["y"], ex[key], rtol=0, atol=1e-14)
        # each token row alone gives the same row (rows are independent)
        for t in range(2):
            part = orc.layer_forward(inp, ex["n_groups"], ex["k"], act, renorm=renorm, rows=[t])
            np.testing.assert_allclose(part["y"][0], ex[key][t], rtol=0, atol=1e-14)


def pin_layer_rows_subset(orc, seed=13):
    """Computing the expert part on a subset of rows gives those rows of the full result
    (tokens are independent in Eq. 1)."""
    rng = np.random.default_rng(seed)
    inp = _rand_layer(rng, 20, 8, 8, 6, 2, orc.SWIGLU, 4, n_shared=1)
    inp["mask"] = np.array([1, 1, 1, 0, 1, 1, 0, 1], np.uint8)
    full = orc.layer_forward(inp, 2, 2, orc.SWIGLU)
    rows = [3, 17, 0, 9]
    part = orc.layer_forward(inp, 2, 2, orc.SWIGLU, rows=rows)
    np.testing.assert_allclose(part["y"], full["y"][rows], rtol=1e-13, atol=1e-14)


# ----------------------------------------------------------- top-group pruning

def _pruning_example():
    ex = golden()["group_pruning"]
    X = np.array(ex["x"])
    Wl = np.array([[_num(v) for v in row] for row in ex["W_local"]])
    Wg = np.array([[_num(v) for v in row] for row in ex["W_global"]])
    return ex, X, Wl, np.array(ex["b_local"]), Wg, np.array(ex["b_global"])


def pin_pruning_golden(orc):
    """Hand-derived g, Top-k, group margins and the rejection of the worked
    pruning example (closed forms)."""
    ex, X, Wl, bl, Wg, bg = _pruning_example()
    K = ex["n_groups"]
    for case in ex["cases"]:
        mask = np.array(case["mask"], np.uint8)
        G = case["top_groups"]
        r = orc.gate_and_route(X, Wl, bl, Wg, bg, mask, K, 1, top_groups=G)
        np.testing.assert_allclose(r["g"], case["g"], rtol=0, atol=1e-12)
        assert r["idx"].tolist() == case["top1"]
        l, m = orc.gate_logits(X, Wl, bl, Wg, bg)
        _, _, gap = orc.group_gate_pruned(l, m, mask.astype(bool), K, G)
        want = [np.inf if v is None else _num(v) for v in case["group_gap"]]
        np.testing.assert_allclose(gap, want, rtol=0, atol=1e-12)
        if case["top2"] is None:
            try:
                orc.gate_and_route(X, Wl, bl, Wg, bg, mask, K, 2, top_groups=G)
            except ValueError:
                pass
            else:
                raise AssertionError("k above the kept groups' candidates must be rejected")
        else:
            r2 = orc.gate_and_route(X, Wl, bl, Wg, bg, mask, K, 2, top_groups=G)
            assert r2["idx"].tolist() == case["top2"]
            np.testing.assert_allclose(r2["w"], np.take_along_axis(np.array(case["g"]), r2["idx"], axis=1),
                                       rtol=0, atol=1e-12)


def pin_pruning_all_groups_is_unpruned(orc, seed=14):
    """Keeping every live group (top_groups >= live groups) is the unpruned gate."""
    rng = np.random.default_rng(seed)
    for (E, K) in [(8, 2), (12, 3), (64, 8)]:
        X, Wl, bl, Wg, bg = _rand_gate(rng, 30, 16, E, K)
        mask = (rng.random(E) < 0.6).astype(np.uint8)
        mask[: E // K] = 0  # one dead group
        mask[E // K] = 1
        allowed = mask.astype(bool)
        l, m = orc.gate_logits(X, Wl, bl, Wg, bg)
        g0, lg0 = orc.group_gate(l, m, allowed, K)
        for G in (K - 1, K):
            g1, lg1, gap = orc.group_gate_pruned(l, m, allowed, K, G)
            np.testing.assert_allclose(g1, g0, rtol=1e-12, atol=1e-15)
            assert np.all(np.isinf(gap))


def pin_pruning_bruteforce(orc, seed=15):
    """Per token, the kept groups are the size-G subset of live groups with the
    largest total p_group (ties to the lexicographically smallest subset), and
    g is scipy's softmax of m over that subset times scipy's softmax of l over
    each kept group's allowed members; Top-k is the brute-force best k-subset
    of the candidates with the lower-index tie rule."""
    rng = np.random.default_rng(seed)
    for (E, K, G, k) in [(8, 4, 2, 3), (12, 4, 1, 2), (6, 3, 2, 3)]:
        T = 40
        X = rng.integers(-2, 3, size=(T, 3)).astype(np.float64)
        Wl = rng.integers(-1, 2, size=(E, 3)).astype(np.float64) * 0.5
        Wg = rng.integers(-1, 2, size=(K, 3)).astype(np.float64) * 0.5
        bl, bg = np.zeros(E), np.zeros(K)
        mask = np.ones(E, np.uint8)
        mask[rng.choice(E, 1)] = 0
        r = orc.gate_and_route(X, Wl, bl, Wg, bg, mask, K, k, top_groups=G)
        gsz = E // K
        live = [j for j in range(K) if mask[j * gsz:(j + 1) * gsz].any()]
        lx, mx = X @ Wl.T + bl, X @ Wg.T + bg
        for t in range(T):
            pg = softmax(mx[t, live])
            best = max(itertools.combinations(range(len(live)), G),
                       key=lambda S: (round(float(sum(pg[list(S)])), 12), [-q for q in S]))
            kept = [live[q] for q in best]
            pg_kept = softmax(mx[t, kept])
            want = np.zeros(E)
            for q, j in enumerate(kept):
                mem = [i for i in range(j * gsz, (j + 1) * gsz) if mask[i]]
                want[mem] = pg_kept[q] * softmax(lx[t, mem])
            np.testing.assert_allclose(r["g"][t], want, rtol=1e-12, atol=1e-15)
            cand = np.flatnonzero(want > 0)
            best_sub = min(itertools.combinations(cand.tolist(), k),
                           key=lambda S: (-round(float(want[list(S)].sum()), 12), S))
            got = r["idx"][t].tolist()
            assert sorted(got) == list(best_sub), (t, got, best_sub)


ALL_PINS = [
    pin_gate_golden, pin_gate_sums_to_one, pin_masked_never_selected, pin_single_group_is_softmax,
    pin_group_factorisation, pin_topk_bruteforce, pin_rejections, pin_route_golden,
    pin_route_invariants, pin_codec_golden, pin_codec_identity, pin_codec_projection,
    pin_ffn_golden, pin_activations_library, pin_ffn_bruteforce, pin_layer_single_expert,
    pin_layer_linearity, pin_layer_codec_golden, pin_layer_rows_subset, pin_layer_pairing_golden,
    pin_pruning_golden, pin_pruning_all_groups_is_unpruned, pin_pruning_bruteforce,
]
