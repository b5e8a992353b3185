"""Boundary-shaped driver of the oracle: one call verifies a batch of draft
trees from logits, draft probabilities and pre-drawn uniforms.

TEST INFRASTRUCTURE ONLY: imported by tests/, the smoke check and the CPU
legs of bench.py, never by the product path.

Inputs follow the statement of the problem in Definition 2 (§3.3) and the
inputs listed by Algorithm 3: the tree, the draft distributions of the
non-leaf nodes and the target distributions of every node.

* M_b(.|X^i) = softmax(logits[i] / T) computed in float64 from the given
  (bf16 or fp32) logit values; the temperature scales the target only
  (Table 4 varies it; the paper does not say more).
* M_s(.|X^i) = draft_probs[i] taken as given (float32 -> float64).
* uniforms[i] (i = 1..N) is the eta of the test of node i; each node is
  tested at most once, so one pre-drawn uniform per node has the same law as
  the fresh draw of Algorithm 3.  uniforms[N+1] draws the bonus token.
* Acceptance is the strict test eta < p (Algorithm 3).
* The bonus token Y is the smallest y with u * W < sum_{x <= y} w(x), where
  w is the accepted node's current M_b and W its total (inverse CDF in
  ascending token order).
"""

import numpy as np

from .traversal import InvalidTree, TraversalState


def softmax_f64(logits_row, temperature):
    """softmax(l / T) in float64 (the plain definition, shifted by the max)."""
    z = np.asarray(logits_row, dtype=np.float64) / np.float64(temperature)
    e = np.exp(z - z.max())
    return e / e.sum()


def inverse_cdf(w, u):
    """Smallest y with u * W < CDF(y); also returns the decision margin
    min(u W - CDF(y-1), CDF(y) - u W) / W."""
    c = np.cumsum(np.asarray(w, dtype=np.float64))
    W = c[-1]
    t = np.float64(u) * W
    y = int(np.searchsorted(c, t, side="right"))
    y = min(y, len(c) - 1)
    lo = c[y - 1] if y > 0 else 0.0
    margin = min(t - lo, c[y] - t) / W
    return y, float(margin), float(W)


def verify_tree(parents, tokens, logits, draft_probs, temperature, uniforms, keep_cdf=False):
    """Traversal Verification of one tree.

    ``logits`` / ``draft_probs`` are [N+1, V] arrays (any float dtype; bf16
    values should arrive already widened to float32), ``uniforms`` is [N+2].
    Returns a dict with the accepted path (node ids, root excluded), tau, the
    bonus token, and the instrumentation used by the parity tests: the rate
    of every tested node at its test, the decision margins, the number of
    S-computations per node and the rows the method had to read.
    """
    parents = np.asarray(parents).astype(np.int64)
    tokens = np.asarray(tokens).astype(np.int64)
    n = len(parents)
    V = logits.shape[1]
    T = float(np.float32(temperature))
    if not T > 0:
        raise ValueError("temperature must be > 0 (the paper's method needs sampling)")
    u = np.asarray(uniforms, dtype=np.float64)

    st = TraversalState(parents, tokens,
                        target_row=lambda i: softmax_f64(logits[i], T),
                        draft_row=lambda i: np.asarray(draft_probs[i], dtype=np.float64),
                        vocab=V)
    node_p = np.full(n, np.nan)
    tests = []
    kappa_at_test = []
    S_at_test = []
    while True:
        leaf = st.first_leaf()
        if leaf == 0:
            accepted = 0
            break
        p = float(st.p[leaf])
        node_p[leaf] = p
        tests.append((leaf, float(u[leaf]), p))
        kappa_at_test.append(max(st.kappa, default=1.0))
        S_at_test.append(st.kappa_S[int(np.argmax(st.kappa))] if st.kappa else float("nan"))
        if u[leaf] < p:
            accepted = leaf
            break
        st.reject(leaf)
    for c in st.pruned:
        node_p[c] = 0.0
    w = st.bonus_weights(accepted)
    y, y_margin, W = inverse_cdf(w, u[n])
    cdf = np.cumsum(np.asarray(w, dtype=np.float64)) if keep_cdf else None
    path = st.path(accepted)
    internal = [i for i in range(n) if st.children[i]]
    return {
        "path": path,
        "tau": len(path),
        "bonus": y,
        "accepted": accepted,
        "node_p": node_p,
        "tests": tests,
        "kappa_at_test": kappa_at_test,
        "S_at_test": S_at_test,
        "test_margin": min((abs(uu - pp) for _, uu, pp in tests), default=np.inf),
        "bonus_margin": y_margin,
        "bonus_total": W,
        "passes": list(st.passes),
        "n_passes": int(sum(st.passes)),
        "rejected_at": [i for i in range(n) if st.passes[i] > 0],
        "internal": internal,
        "leaf_row_read": accepted not in st.mb,
        "pruned": list(st.pruned),
        "degenerate": st.degenerate,
        "bonus_u": float(u[n]),
        "bonus_cdf": cdf,
    }


def algorithmic_bytes(result, vocab, logit_bytes):
    """Bytes the method must read for one tree under the eager initialisation
    of Algorithm 3: one target row per internal node, one draft row per node at
    which S was computed at least once, and the accepted leaf's target row."""
    n_int = len(result["internal"])
    r = len(result["rejected_at"])
    leaf = 1 if result["leaf_row_read"] else 0
    return vocab * (n_int * logit_bytes + r * 4 + leaf * logit_bytes)


def verify_batch(parents, tokens, logits, draft_probs, temperature, uniforms,
                 trees=None, keep_cdf=False, tree_fn=None):
    """Batch driver: arrays [B, N+1], [B, N+1], [B, N+1, V], [B, N+1, V],
    scalar, [B, N+2].  Invalid trees get tau = -1, bonus = -1 and an all -1
    path, the same marking the library uses.  ``trees`` restricts the work to a
    subset of tree indices (others are left marked -2).  ``tree_fn`` is the
    per-tree verifier (default: Traversal Verification, ``verify_tree``)."""
    tree_fn = verify_tree if tree_fn is None else tree_fn
    parents = np.asarray(parents)
    B, n = parents.shape
    out_path = np.full((B, max(n - 1, 0)), -1, dtype=np.int32)
    out_tau = np.full(B, -2, dtype=np.int32)
    out_bonus = np.full(B, -2, dtype=np.int32)
    details = {}
    idx = range(B) if trees is None else trees
    for b in idx:
        try:
            r = tree_fn(parents[b], tokens[b], logits[b], draft_probs[b],
                        temperature, uniforms[b], keep_cdf=keep_cdf)
        except InvalidTree as e:
            out_tau[b] = -1
            out_bonus[b] = -1
            details[b] = {"invalid": str(e)}
            continue
        out_tau[b] = r["tau"]
        out_bonus[b] = r["bonus"]
        out_path[b, :r["tau"]] = r["path"]
        details[b] = r
    return out_path, out_tau, out_bonus, details
