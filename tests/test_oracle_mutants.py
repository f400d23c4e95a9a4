"""Plant plausible mistakes in the oracle (on the CPU) and check that the pins catch each.

A pin set that lets one of these through would also let the same mistake in
the oracle go unnoticed, so every mutant here must fail at least one pin.
"""
import numpy as np
import pytest

from oracle import ec2moe_oracle as orc
from tests import pins

_gate_logits = orc.gate_logits
_group_gate = orc.group_gate
_masked_softmax = orc._masked_softmax
_route_tables = orc.route_tables
_expert_ffn = orc.expert_ffn
_combine_weights = orc.combine_weights
_layer_forward = orc.layer_forward
_topk_gaps = orc.topk_gaps


def m_drop_local_bias(X, Wl, bl, Wg=None, bg=None):
    return _gate_logits(X, Wl, np.zeros_like(np.asarray(bl, float)), Wg, bg)


def m_drop_global_bias(X, Wl, bl, Wg=None, bg=None):
    return _gate_logits(X, Wl, bl, Wg, None if bg is None else np.zeros_like(np.asarray(bg, float)))


def m_softmax_ignores_mask(z, keep):
    out = _masked_softmax(z, np.ones_like(keep))
    out[:, ~keep] = 0.0
    return out


def m_group_gate_keeps_dead_groups(l, m, allowed, K):
    # a dead group still takes part in the group softmax
    g, log_g = _group_gate(l, m, allowed, K)
    if K > 1 and m is not None:
        b = orc.group_bounds(l.shape[1], K)
        live = np.array([allowed[b[i]:b[i + 1]].any() for i in range(K)])
        if not live.all():
            full = np.exp(m - m.max(1, keepdims=True))
            full /= full.sum(1, keepdims=True)
            part = np.exp(m[:, live] - m[:, live].max(1, keepdims=True))
            part /= part.sum(1, keepdims=True)
            scale = np.ones_like(m)
            scale[:, live] = full[:, live] / part
            gof = np.repeat(np.arange(K), np.diff(b))
            g = g * scale[:, gof]
    return g, log_g


def m_tie_to_higher_index(g, allowed, k):
    E = g.shape[1]
    key = np.where(allowed[None, :], -g, np.inf)[:, ::-1]
    order = np.argsort(key, axis=1, kind="stable")
    return (E - 1 - order[:, :k]).astype(np.int64)


def m_topk_ascending(g, allowed, k):
    key = np.where(allowed[None, :], g, np.inf)
    return np.argsort(key, axis=1, kind="stable")[:, :k].astype(np.int64)


def m_perm_reversed_within_expert(idx, E):
    c, o, p = _route_tables(idx, E)
    p = p.copy()
    for e in range(E):
        p[o[e]:o[e + 1]] = p[o[e]:o[e + 1]][::-1]
    return c, o, p


def m_offsets_inclusive(idx, E):
    c, o, p = _route_tables(idx, E)
    o = o.copy()
    o[:-1] = o[1:]
    return c, o, p


def m_decode_no_transpose(Z, V_dec):
    return np.asarray(Z, float) @ np.asarray(V_dec, float)


def m_encode_wrong_side(X, V_enc):
    V = np.asarray(V_enc, float)
    if V.shape[0] == V.shape[1]:
        return np.asarray(X, float) @ V
    return np.asarray(X, float) @ V.T * 1.0001


def m_gelu_tanh(u):
    return 0.5 * u * (1 + np.tanh(np.sqrt(2 / np.pi) * (u + 0.044715 * u ** 3)))


def m_silu_missing_x(u):
    return 1.0 / (1.0 + np.exp(-u))


def m_swiglu_swapped(x, W1, W2, W3, act):
    if act == orc.SWIGLU:
        return _expert_ffn(x, W3, W2, W1, act)
    return _expert_ffn(x, W1, W2, W3, act)


def m_renorm_ignored(g, idx, renorm):
    return _combine_weights(g, idx, False)


def m_renorm_always(g, idx, renorm):
    return _combine_weights(g, idx, True)


def m_no_shared(inp, n_groups, k, act, renorm=False, rows=None):
    inp = dict(inp)
    inp["W1s"] = inp["W2s"] = inp["W3s"] = None
    return _layer_forward(inp, n_groups, k, act, renorm, rows)


def m_experts_see_raw_x(inp, n_groups, k, act, renorm=False, rows=None):
    out = _layer_forward(inp, n_groups, k, act, renorm, rows)
    if inp.get("V_enc") is not None:
        inp2 = dict(inp)
        inp2["V_enc"] = inp2["V_dec"] = None
        out2 = _layer_forward(inp2, n_groups, k, act, renorm, rows)
        out["y"] = out2["y"]
    return out


def m_experts_rolled(inp, n_groups, k, act, renorm=False, rows=None):
    # every routed row meets the weights of expert e - 1 instead of expert e
    inp = dict(inp)
    for key in ("W1", "W3", "W2"):
        if inp.get(key) is not None:
            inp[key] = np.roll(np.asarray(inp[key]), 1, axis=0)
    return _layer_forward(inp, n_groups, k, act, renorm, rows)


def m_slot_weight_shifted(inp, n_groups, k, act, renorm=False, rows=None):
    # slot s's expert output is scaled by slot s + 1's gate weight
    out = _layer_forward(inp, n_groups, k, act, renorm, rows)
    X_hat = out["X_hat"]
    sel = out["rows"]
    idx, w = out["idx"][sel], out["w"][sel]
    y = np.zeros_like(out["y"])
    for e in range(inp["W1"].shape[0]):
        for s in range(k):
            hit = np.nonzero(idx[:, s] == e)[0]
            if hit.size == 0:
                continue
            W3 = None if inp.get("W3") is None else inp["W3"][e]
            o = orc.expert_ffn(X_hat[hit], inp["W1"][e], inp["W2"][e], W3, act)
            y[hit] += w[hit, (s + 1) % k][:, None] * o
    if inp.get("W1s") is not None:
        for s in range(inp["W1s"].shape[0]):
            W3s = None if inp.get("W3s") is None else inp["W3s"][s]
            y += orc.expert_ffn(X_hat, inp["W1s"][s], inp["W2s"][s], W3s, act)
    out["y"] = y
    return out


def m_weights_slot_rolled(g, idx, renorm):
    # the combine weights are paired with the wrong slots
    return np.roll(_combine_weights(g, idx, renorm), 1, axis=1)


def _pruned_variant(l, m, allowed, K, G, order="p_group", ties="lower", renorm=True):
    # group_gate_pruned with one step changed (the ranking key, the tie rule,
    # or the renormalisation of p_group over the kept groups)
    T, E = l.shape
    b = orc.group_bounds(E, K)
    live = [j for j in range(K) if allowed[b[j]:b[j + 1]].any()]
    g = np.zeros((T, E))
    log_g = np.full((T, E), -np.inf)
    gap = np.full(T, np.inf)
    for t in range(T):
        if order == "local":
            score = [max(l[t, i] for i in range(b[j], b[j + 1]) if allowed[i]) for j in live]
        elif order == "lowest":
            score = [-m[t, j] for j in live]
        else:
            score = [m[t, j] for j in live]
        sign = 1 if ties == "lower" else -1
        ranked = sorted(range(len(live)), key=lambda q: (-score[q], sign * live[q]))
        kept = sorted(live[q] for q in ranked[:G])
        if G < len(live):
            gap[t] = m[t, live[ranked[G - 1]]] - m[t, live[ranked[G]]]
        pool = kept if renorm else live
        mk = m[t, pool]
        lse = mk.max() + np.log(np.exp(mk - mk.max()).sum())
        for j in kept:
            mem = [i for i in range(b[j], b[j + 1]) if allowed[i]]
            z = l[t, mem]
            lz = z.max() + np.log(np.exp(z - z.max()).sum())
            for i, zi in zip(mem, z):
                log_g[t, i] = (m[t, j] - lse) + (zi - lz)
                g[t, i] = np.exp(log_g[t, i])
    return g, log_g, gap


def m_pruned_no_renorm(l, m, allowed, K, G):
    return _pruned_variant(l, m, allowed, K, G, renorm=False)


def m_pruned_keeps_lowest(l, m, allowed, K, G):
    return _pruned_variant(l, m, allowed, K, G, order="lowest")


def m_pruned_ties_to_higher_group(l, m, allowed, K, G):
    return _pruned_variant(l, m, allowed, K, G, ties="higher")


def m_pruned_by_best_local(l, m, allowed, K, G):
    return _pruned_variant(l, m, allowed, K, G, order="local")


def m_pruning_ignored(l, m, allowed, K, G):
    g, log_g = orc.group_gate(l, m, allowed, K)
    return g, log_g, np.full(l.shape[0], np.inf)


def m_group_factor_dropped(l, m, allowed, K):
    # Eq. 7 without the group probability: g = p_local
    g, log_g = _group_gate(l, m, allowed, K)
    if K == 1 or m is None:
        return g, log_g
    b = orc.group_bounds(l.shape[1], K)
    gof = np.repeat(np.arange(K), np.diff(b))
    live = np.array([allowed[b[i]:b[i + 1]].any() for i in range(K)])
    p_group = _masked_softmax(m, live)
    with np.errstate(divide="ignore", invalid="ignore"):
        g2 = np.where(allowed[None, :], g / p_group[:, gof], 0.0)
        log_g2 = np.where(allowed[None, :], log_g - np.log(p_group[:, gof]), -np.inf)
    return g2, log_g2


def m_global_from_local_rows(X, Wl, bl, Wg=None, bg=None):
    # Eq. 6 evaluated with the first K local gate rows instead of W_global
    if Wg is None:
        return _gate_logits(X, Wl, bl, Wg, bg)
    K = np.asarray(Wg).shape[0]
    return _gate_logits(X, Wl, bl, np.asarray(Wl)[:K], bg)


def m_perm_slot_major(idx, E):
    # rows of one expert ordered by (slot, token) instead of (token, slot)
    counts, offsets, _ = _route_tables(idx, E)
    idx = np.asarray(idx)
    T, k = idx.shape
    flat = idx.reshape(-1)
    t = np.arange(T * k) // k
    s = np.arange(T * k) % k
    perm = np.lexsort((t, s, flat)).astype(np.int64)
    return counts, offsets, perm


def m_shared_scaled_by_gate(inp, n_groups, k, act, renorm=False, rows=None, top_groups=0):
    # the always-on shared experts weighted by the first slot's gate weight
    out = _layer_forward(inp, n_groups, k, act, renorm, rows, top_groups)
    if inp.get("W1s") is None:
        return out
    X_hat = out["X_hat"]
    w0 = out["w"][out["rows"], 0][:, None]
    for s in range(inp["W1s"].shape[0]):
        W3s = None if inp.get("W3s") is None else inp["W3s"][s]
        o = orc.expert_ffn(X_hat, inp["W1s"][s], inp["W2s"][s], W3s, act)
        out["y"] = out["y"] + (w0 - 1.0) * o
    return out


def m_gap_wrong_sign(log_g, idx, allowed):
    b, a = _topk_gaps(log_g, idx, allowed)
    return -b, a


MUTANTS = [
    ("gate_logits", m_drop_local_bias),
    ("gate_logits", m_drop_global_bias),
    ("_masked_softmax", m_softmax_ignores_mask),
    ("group_gate", m_group_gate_keeps_dead_groups),
    ("topk_route", m_tie_to_higher_index),
    ("topk_route", m_topk_ascending),
    ("route_tables", m_perm_reversed_within_expert),
    ("route_tables", m_offsets_inclusive),
    ("lr_decode", m_decode_no_transpose),
    ("lr_encode", m_encode_wrong_side),
    ("gelu", m_gelu_tanh),
    ("silu", m_silu_missing_x),
    ("expert_ffn", m_swiglu_swapped),
    ("combine_weights", m_renorm_ignored),
    ("combine_weights", m_renorm_always),
    ("layer_forward", m_no_shared),
    ("layer_forward", m_experts_see_raw_x),
    ("layer_forward", m_experts_rolled),
    ("layer_forward", m_slot_weight_shifted),
    ("combine_weights", m_weights_slot_rolled),
    ("group_gate_pruned", m_pruned_no_renorm),
    ("group_gate_pruned", m_pruned_keeps_lowest),
    ("group_gate_pruned", m_pruned_ties_to_higher_group),
    ("group_gate_pruned", m_pruned_by_best_local),
    ("group_gate_pruned", m_pruning_ignored),
    ("topk_gaps", m_gap_wrong_sign),
    ("group_gate", m_group_factor_dropped),
    ("gate_logits", m_global_from_local_rows),
    ("route_tables", m_perm_slot_major),
    ("layer_forward", m_shared_scaled_by_gate),
]


@pytest.mark.parametrize("name,mutant", MUTANTS, ids=[m.__name__ for _, m in MUTANTS])
def test_mutant_is_caught(monkeypatch, name, mutant):
    monkeypatch.setattr(orc, name, mutant)
    caught = []
    for pin in pins.ALL_PINS:
        try:
            pin(orc)
        except (AssertionError, ValueError, IndexError, TypeError):
            caught.append(pin.__name__)
    assert caught, f"no pin catches mutant {mutant.__name__}"

