"""fp64 CPU oracle for the EC²MoE MoE-layer forward (arXiv 2508.06024).

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this module.  It
shares no code with the CUDA path and never calls it.

Every function is the plain definition of one step, written in float64 with
numpy; a matrix product, a sort or ``erf`` are used as library primitives and
nothing is blocked, fused or reordered.  Inputs are the stored (bf16- or
fp32-rounded) tensors widened exactly to float64.

Steps and the passages they follow:

* ``allowed_experts``   - Eq. 4, the local candidate set E_local (here an
  input mask; the capability function H and matching function f of Eq. 3-4
  are not specified by the paper).
* ``gate_logits``       - the affine maps inside Eq. 5 (W_k x + b_k, groups
  stacked into one [E, d] matrix) and Eq. 6 (W_global x + b_global).
* ``group_gate``        - Eq. 5 (per-group softmax), Eq. 6 (group softmax) and
  Eq. 7 (g_i = p_group^(k) * p_local,i^(k)), restricted to allowed experts.
* ``group_gate_pruned`` - the hierarchical use of Eq. 5-7 with top-group
  pruning: Eq. 6 first, then Eq. 5 only inside the top groups, then Eq. 7
  (the "lightweight" evaluation the group gate section motivates).
* ``topk_route``        - Top-k selection (Top-1 in the evaluation setup),
  ties to the lower expert index.
* ``route_tables``      - per-expert histogram, exclusive scan and the stable
  expert-major permutation of (token, slot) pairs.
* ``lr_encode`` / ``lr_decode`` - the low-rank encoder Z = U^T X V and decoder
  X_hat = U_hat Z V_hat^T of the end-cloud codec, with the token-side
  projections U = U_hat = I on a [tokens, d_model] activation matrix.
* ``expert_ffn``        - one expert E_i of Eq. 1 (GELU or SwiGLU FFN, no bias).
* ``layer_forward``     - Eq. 1, y = sum_i G(x)_i E_i(x), over the top-k
  experts with G = g (optionally renormalised over the top-k), plus
  always-on shared experts.

Readings where the paper is silent (each also listed in the design notes):
masked experts are never selected; a group without allowed members drops out
of the group softmax; K = 1 means p_group = 1; GELU is the exact erf form;
the codec is one-sided on the d_model axis.
"""

from __future__ import annotations

from typing import Dict, Optional, Sequence

import numpy as np
from scipy.special import erf

GELU = 0
SWIGLU = 1


def group_bounds(E: int, n_groups: int) -> np.ndarray:
    """Contiguous equal-size groups: group k owns experts [k*E/K, (k+1)*E/K).

    Eq. 5 splits the M experts into K groups of M_k experts; the paper does not
    say how, so the groups are contiguous and of equal size.
    """
    if n_groups < 1 or E % n_groups != 0:
        raise ValueError("E must be a positive multiple of n_groups")
    size = E // n_groups
    return np.arange(0, E + 1, size, dtype=np.int64)


def allowed_experts(mask: np.ndarray, k: int) -> np.ndarray:
    """Eq. 4: the local candidate set as a boolean vector.

    Raises ValueError when no expert is allowed or fewer than k are.
    """
    allowed = np.asarray(mask).astype(bool)
    n = int(allowed.sum())
    if n == 0:
        raise ValueError("all experts masked")
    if n < k:
        raise ValueError("fewer allowed experts than k")
    return allowed


def gate_logits(X, W_local, b_local, W_global=None, b_global=None):
    """Eq. 5 and Eq. 6 pre-softmax: l = X W_local^T + b_local, m = X W_global^T + b_global.

    X [T, d]; W_local [E, d] (the group matrices W_k stacked in group order);
    W_global [K, d] or None when K = 1.  Returns (l [T, E], m [T, K] or None).
    """
    X = np.asarray(X, dtype=np.float64)
    l = X @ np.asarray(W_local, dtype=np.float64).T + np.asarray(b_local, dtype=np.float64)
    m = None
    if W_global is not None:
        m = X @ np.asarray(W_global, dtype=np.float64).T + np.asarray(b_global, dtype=np.float64)
    return l, m


def _masked_softmax(z: np.ndarray, keep: np.ndarray) -> np.ndarray:
    """Softmax of each row of z over the columns where keep is True; 0 elsewhere."""
    out = np.zeros_like(z)
    if not keep.any():
        return out
    zk = z[:, keep]
    zk = zk - zk.max(axis=1, keepdims=True)
    e = np.exp(zk)
    out[:, keep] = e / e.sum(axis=1, keepdims=True)
    return out


def group_gate(l: np.ndarray, m: Optional[np.ndarray], allowed: np.ndarray, n_groups: int):
    """Eq. 5-7 on allowed experts.

    p_local: softmax of l over the allowed members of each group (Eq. 5).
    p_group: softmax of m over the groups that keep at least one allowed
    member (Eq. 6); 1 when K = 1.
    g_i = p_group[group(i)] * p_local[i] (Eq. 7); g_i = 0 for masked i.
    Returns (g [T, E], log_g [T, E] with -inf on masked experts).
    """
    T, E = l.shape
    bounds = group_bounds(E, n_groups)
    p_local = np.zeros((T, E))
    log_p_local = np.full((T, E), -np.inf)
    group_live = np.zeros(n_groups, dtype=bool)
    for k in range(n_groups):
        lo, hi = bounds[k], bounds[k + 1]
        keep = allowed[lo:hi]
        if not keep.any():
            continue
        group_live[k] = True
        lk = l[:, lo:hi]
        p_local[:, lo:hi] = _masked_softmax(lk, keep)
        zk = lk[:, keep]
        lse = zk.max(axis=1, keepdims=True) + np.log(np.exp(zk - zk.max(axis=1, keepdims=True)).sum(axis=1, keepdims=True))
        sub = np.full(lk.shape, -np.inf)
        sub[:, keep] = lk[:, keep] - lse
        log_p_local[:, lo:hi] = sub
    if n_groups == 1:
        p_group = np.ones((T, 1))
        log_p_group = np.zeros((T, 1))
    else:
        if m is None:
            raise ValueError("global gate required when n_groups > 1")
        p_group = _masked_softmax(m, group_live)
        mk = m[:, group_live]
        lse = mk.max(axis=1, keepdims=True) + np.log(np.exp(mk - mk.max(axis=1, keepdims=True)).sum(axis=1, keepdims=True))
        log_p_group = np.full(m.shape, -np.inf)
        log_p_group[:, group_live] = m[:, group_live] - lse
    group_of = np.repeat(np.arange(n_groups), np.diff(bounds))
    g = p_group[:, group_of] * p_local
    log_g = log_p_group[:, group_of] + log_p_local
    g[:, ~allowed] = 0.0
    log_g[:, ~allowed] = -np.inf
    return g, log_g


def pruned_candidate_floor(allowed: np.ndarray, n_groups: int, top_groups: int) -> int:
    """Fewest allowed experts that any choice of ``top_groups`` live groups holds
    (the sum of the smallest per-group allowed counts); Top-k needs k of them."""
    E = allowed.shape[0]
    b = group_bounds(E, n_groups)
    sizes = sorted(int(allowed[b[j]:b[j + 1]].sum()) for j in range(n_groups) if allowed[b[j]:b[j + 1]].any())
    return int(sum(sizes[:top_groups]))


def group_gate_pruned(l: np.ndarray, m: np.ndarray, allowed: np.ndarray, n_groups: int, top_groups: int):
    """Eq. 5-7 evaluated hierarchically with top-group pruning.

    Per token, in the paper's order:
      1. Eq. 6: the group probabilities p_group = softmax of m over the live
         groups (those with an allowed member).
      2. Keep the ``top_groups`` live groups with the largest p_group (ties to
         the lower group index); the others are pruned for this token.
      3. Eq. 5 only inside the kept groups: p_local = softmax of l over the
         allowed members of each kept group.
      4. Eq. 7: g_i = p_group'^(k) * p_local,i, where p_group' is p_group
         renormalised over the kept groups, so that the gate still sums to 1
         over its candidates as Eq. 1 requires.  Experts of pruned groups (and
         masked experts) get g = 0 and log g = -inf.
    ``top_groups`` >= the number of live groups keeps every live group, which
    is ``group_gate`` itself.  Returns (g [T, E], log_g [T, E], group_gap [T]):
    group_gap is the margin in m between the last kept group and the best
    pruned one (+inf when nothing is pruned), used to exclude near-ties of the
    group decision from exact checks.
    """
    T, E = l.shape
    bounds = group_bounds(E, n_groups)
    live = [j for j in range(n_groups) if allowed[bounds[j]:bounds[j + 1]].any()]
    g = np.zeros((T, E))
    log_g = np.full((T, E), -np.inf)
    group_gap = np.full(T, np.inf)
    for t in range(T):
        # step 1: Eq. 6 over the live groups
        p_group = np.exp(m[t, live] - m[t, live].max())
        p_group /= p_group.sum()
        # step 2: the top groups by p_group, ties to the lower group index
        ranked = sorted(range(len(live)), key=lambda q: (-p_group[q], live[q]))
        kept = sorted(live[q] for q in ranked[:top_groups])
        if top_groups < len(live):
            group_gap[t] = m[t, live[ranked[top_groups - 1]]] - m[t, live[ranked[top_groups]]]
        # step 4's renormalised group probabilities over the kept groups
        mk = m[t, kept]
        lse_kept = mk.max() + np.log(np.exp(mk - mk.max()).sum())
        for j in kept:
            lo, hi = bounds[j], bounds[j + 1]
            members = [i for i in range(lo, hi) if allowed[i]]
            # step 3: Eq. 5 inside the kept group
            z = l[t, members]
            lse_j = z.max() + np.log(np.exp(z - z.max()).sum())
            log_pg = m[t, j] - lse_kept
            for i, zi in zip(members, z):
                log_g[t, i] = log_pg + (zi - lse_j)
                g[t, i] = np.exp(log_g[t, i])
    return g, log_g, group_gap


def topk_route(g: np.ndarray, allowed: np.ndarray, k: int):
    """Top-k experts per token by g, ties to the lower expert index.

    A stable sort of (-g) keeps equal keys in index order, which is exactly the
    tie rule; masked experts sort last.  Returns idx [T, k] int64 in slot
    order (largest g first).
    """
    key = np.where(allowed[None, :], -g, np.inf)
    order = np.argsort(key, axis=1, kind="stable")
    return order[:, :k].astype(np.int64)


def topk_gaps(log_g: np.ndarray, idx: np.ndarray, allowed: np.ndarray):
    """Decision margins in log g, used to exclude near-ties from exact checks.

    Returns (boundary_gap [T], adjacent_gaps [T, k-1]):
    boundary_gap = log g of slot k-1 minus the best log g outside the top-k
    (+inf when every allowed expert is selected); adjacent_gaps[:, j] =
    log g of slot j minus slot j+1.
    """
    T, E = log_g.shape
    k = idx.shape[1]
    rows = np.arange(T)[:, None]
    sel = log_g[rows, idx]
    rest = log_g.copy()
    rest[:, ~allowed] = -np.inf
    rest[rows, idx] = -np.inf
    best_rest = rest.max(axis=1)
    boundary = sel[:, -1] - best_rest
    adjacent = sel[:, :-1] - sel[:, 1:]
    return boundary, adjacent


def combine_weights(g: np.ndarray, idx: np.ndarray, renorm: bool) -> np.ndarray:
    """Gate weight of each (token, slot): G(x)_i = g_i, or g_i / sum_topk g when renormalised."""
    w = np.take_along_axis(g, idx, axis=1)
    if renorm:
        w = w / w.sum(axis=1, keepdims=True)
    return w


def route_tables(idx: np.ndarray, E: int):
    """Histogram, exclusive scan and stable expert-major permutation.

    counts[e] = #{(t, s): idx[t, s] = e}; offsets = exclusive prefix sum of
    counts (length E + 1); perm[p] = t * k + s for the p-th row in expert-major
    order, rows of one expert in increasing (t, s).
    """
    flat = np.asarray(idx).reshape(-1)
    counts = np.bincount(flat, minlength=E).astype(np.int64)
    offsets = np.zeros(E + 1, dtype=np.int64)
    offsets[1:] = np.cumsum(counts)
    perm = np.argsort(flat, kind="stable").astype(np.int64)
    return counts, offsets, perm


def lr_encode(X: np.ndarray, V_enc: np.ndarray) -> np.ndarray:
    """Codec encoder Z = U^T X V with U = I on the token axis and V = V_enc^T: Z = X V_enc^T.

    X [T, d], V_enc [r, d] -> Z [T, r].
    """
    return np.asarray(X, dtype=np.float64) @ np.asarray(V_enc, dtype=np.float64).T


def lr_decode(Z: np.ndarray, V_dec: np.ndarray) -> np.ndarray:
    """Codec decoder X_hat = U_hat Z V_hat^T with U_hat = I and V_hat = V_dec: X_hat = Z V_dec^T.

    Z [T, r], V_dec [d, r] -> X_hat [T, d].
    """
    return np.asarray(Z, dtype=np.float64) @ np.asarray(V_dec, dtype=np.float64).T


def gelu(u: np.ndarray) -> np.ndarray:
    """GELU(u) = u * Phi(u) = u/2 * (1 + erf(u / sqrt 2)) (exact form)."""
    return 0.5 * u * (1.0 + erf(u / np.sqrt(2.0)))


def silu(u: np.ndarray) -> np.ndarray:
    """SiLU(u) = u / (1 + exp(-u))."""
    return u / (1.0 + np.exp(-u))


def expert_ffn(x: np.ndarray, W1: np.ndarray, W2: np.ndarray, W3: Optional[np.ndarray], act: int) -> np.ndarray:
    """One expert FFN E_i of Eq. 1 on rows x [n, d].

    GELU:   W2 GELU(W1 x)        (W1 [f, d], W2 [d, f])
    SwiGLU: W2 (SiLU(W1 x) * (W3 x))  (W3 [f, d])
    """
    x = np.asarray(x, dtype=np.float64)
    u = x @ np.asarray(W1, dtype=np.float64).T
    if act == GELU:
        h = gelu(u)
    elif act == SWIGLU:
        h = silu(u) * (x @ np.asarray(W3, dtype=np.float64).T)
    else:
        raise ValueError("unknown activation")
    return h @ np.asarray(W2, dtype=np.float64).T


def gate_and_route(X, W_local, b_local, W_global, b_global, mask, n_groups: int, k: int, renorm: bool = False,
                   top_groups: int = 0):
    """Steps 1-3 for all tokens: mask, group gate, top-k, tables and margins.

    ``top_groups`` > 0 (with n_groups > 1) applies top-group pruning
    (``group_gate_pruned``); k must then not exceed the allowed experts the
    fewest-member choice of top_groups live groups holds.  With pruning the
    boundary margin also covers the group decision (the smaller of the two)."""
    allowed = allowed_experts(mask, k)
    l, m = gate_logits(X, W_local, b_local, W_global, b_global)
    pruned = top_groups > 0 and n_groups > 1
    if pruned:
        if pruned_candidate_floor(allowed, n_groups, top_groups) < k:
            raise ValueError("fewer allowed experts in the kept groups than k")
        g, log_g, group_gap = group_gate_pruned(l, m, allowed, n_groups, top_groups)
        cand = np.isfinite(log_g)
        idx = np.argsort(np.where(cand, -g, np.inf), axis=1, kind="stable")[:, :k].astype(np.int64)
    else:
        g, log_g = group_gate(l, m, allowed, n_groups)
        idx = topk_route(g, allowed, k)
    w = combine_weights(g, idx, renorm)
    counts, offsets, perm = route_tables(idx, l.shape[1])
    boundary, adjacent = topk_gaps(log_g, idx, allowed)
    if pruned:
        boundary = np.minimum(boundary, group_gap)
    return dict(allowed=allowed, l=l, m=m, g=g, log_g=log_g, idx=idx, w=w, counts=counts,
                offsets=offsets, perm=perm, gap_boundary=boundary, gap_adjacent=adjacent)


def layer_forward(inp: Dict[str, np.ndarray], n_groups: int, k: int, act: int, renorm: bool = False,
                  rows: Optional[Sequence[int]] = None, top_groups: int = 0) -> Dict[str, np.ndarray]:
    """The whole MoE-layer forward (Eq. 1 with the Eq. 4-7 gate and the codec).

    ``inp`` holds float64 arrays: X, W_local, b_local, W_global, b_global,
    mask, W1, W3, W2, W1s, W3s, W2s, V_enc, V_dec (absent parts None).
    The gate sees X; the experts see the decoded X_hat (X when no codec).
    ``rows`` restricts the expert/combine part to those token rows (the gate
    and routing always cover every token, since the histogram needs them all).
    ``top_groups`` > 0 selects the pruned group gate (``group_gate_pruned``).
    Returns the routing results plus Z, X_hat and y for the chosen rows.
    """
    X = np.asarray(inp["X"], dtype=np.float64)
    r = gate_and_route(X, inp["W_local"], inp["b_local"], inp.get("W_global"), inp.get("b_global"),
                       inp["mask"], n_groups, k, renorm, top_groups)
    sel = np.arange(X.shape[0]) if rows is None else np.asarray(rows, dtype=np.int64)
    Xs = X[sel]
    if inp.get("V_enc") is not None:
        Z = lr_encode(Xs, inp["V_enc"])
        X_hat = lr_decode(Z, inp["V_dec"])
    else:
        Z = None
        X_hat = Xs
    d = X.shape[1]
    y = np.zeros((len(sel), d))
    idx = r["idx"][sel]
    w = r["w"][sel]
    E = inp["W1"].shape[0]
    for e in range(E):
        for s in range(k):
            hit = np.nonzero(idx[:, s] == e)[0]
            if hit.size == 0:
                continue
            W3 = None if inp.get("W3") is None else inp["W3"][e]
            o = expert_ffn(X_hat[hit], inp["W1"][e], inp["W2"][e], W3, act)
            y[hit] += w[hit, s][:, None] * o
    if inp.get("W1s") is not None:
        for s in range(inp["W1s"].shape[0]):
            W3s = None if inp.get("W3s") is None else inp["W3s"][s]
            y += expert_ffn(X_hat, inp["W1s"][s], inp["W2s"][s], W3s, act)
    r.update(rows=sel, Z=Z, X_hat=X_hat, y=y)
    return r
