"""Draft-side sampling of a token tree (Definition 1): the children of every
node are drawn from the node's draft distribution M_s(.|X^i) without
replacement, in child-index order -- literal and slow.

TEST INFRASTRUCTURE ONLY: imported by tests/, the smoke check and the CPU
legs of bench.py, never by the product path.

Each child c of node i takes one pre-drawn uniform u[c] in [0, 1) and is drawn
by inverse CDF, in ascending token order, from M_s(.|X^i) with the tokens of
the earlier children of i removed (Definition 1 draws siblings without
replacement; the verification takes the children in index order, so they
are drafted in that order):

    q'(x) = q(x) for x not yet drawn among c's earlier siblings, else 0,
    W     = sum_x q'(x),
    token = the smallest y with  u[c] * W < sum_{x <= y} q'(x).

Renormalising q' by W and comparing with u[c] is the same as comparing
u[c] * W with the unnormalised cumulative sums, so no division is done.  A
token with q'(y) = 0 is never drawn (the cumulative sum does not grow there).
If no mass is left (W = 0: more children than tokens of positive draft
probability), the child and every later sibling get -1.  If rounding leaves
u[c] * W at or above the last cumulative sum, the last token of positive
mass is taken.

Generic over float (float64 arithmetic on the given values) and
fractions.Fraction (exact), so the pins can probe interval boundaries
exactly.
"""

from fractions import Fraction

import numpy as np


def draw_without_replacement(q, removed, u):
    """One inverse-CDF draw from q with the tokens in ``removed`` taken out.
    Returns (token, W) with token -1 when no mass is left."""
    if not isinstance(u, Fraction):
        t, W, _ = draw_float(q, removed, u)
        return t, W
    removed = set(removed)
    qp = [Fraction(0) if x in removed else q[x] for x in range(len(q))]
    W = sum(qp, Fraction(0))
    if not W > 0:
        return -1, W
    target = u * W
    cdf = Fraction(0)
    last = -1
    for y, m in enumerate(qp):
        if m > 0:
            last = y
        cdf = cdf + m
        if target < cdf:
            return y, W
    return last, W


def draw_float(q, removed, u):
    """The same draw in float64 (numpy's sequential cumulative sum; the
    smallest y with u W < CDF(y) is searchsorted(side='right')).  Returns
    (token, W, margin), margin = distance of u W from the nearer cumulative
    step bounding the token, relative to W."""
    qp = np.array(q, dtype=np.float64)
    for x in removed:
        if x >= 0:
            qp[x] = 0.0
    cdf = np.cumsum(qp)
    W = float(cdf[-1]) if len(cdf) else 0.0
    if not W > 0:
        return -1, W, np.inf
    target = float(u) * W
    y = int(np.searchsorted(cdf, target, side="right"))
    if y >= len(qp):
        y = int(np.flatnonzero(qp)[-1])
    lo = float(cdf[y - 1]) if y > 0 else 0.0
    margin = min(abs(target - lo), abs(float(cdf[y]) - target)) / W
    return y, W, margin


def sample_children(q, k, uniforms):
    """k children of one node, in order: child j uses uniforms[j]."""
    out = []
    for j in range(k):
        if out and out[-1] < 0:
            out.append(-1)
            continue
        t, _ = draw_without_replacement(q, out, uniforms[j])
        out.append(t)
    return out


def valid_tree(parents):
    """parents[0] = -1 and parents[c] in [0, c) for c >= 1."""
    return int(parents[0]) == -1 and all(0 <= int(parents[c]) < c
                                         for c in range(1, len(parents)))


def sample_tree(parents, drafts, uniforms, margins=None):
    """Tokens [N+1] of one tree: node c >= 1 is drawn from drafts[parents[c]]
    with the tokens of its earlier siblings removed, using uniforms[c]; entry
    0 (the root's own token, not drafted here) is 0.  An invalid parent array
    gives -1 for every node c >= 1.  ``margins``, if a list, receives each
    node's draw margin (float draws only; inf where no draw was made)."""
    n = len(parents)
    tokens = [0] * n
    if margins is not None:
        margins[:] = [np.inf] * n
    if not valid_tree(parents):
        return [0] + [-1] * (n - 1)
    kids = {}
    for c in range(1, n):
        p = int(parents[c])
        earlier = kids.setdefault(p, [])
        if earlier and tokens[earlier[-1]] < 0:
            tokens[c] = -1
        elif margins is not None:
            tokens[c], _, margins[c] = draw_float(drafts[p], [tokens[j] for j in earlier],
                                                  uniforms[c])
        else:
            tokens[c], _ = draw_without_replacement(drafts[p], [tokens[j] for j in earlier],
                                                    uniforms[c])
        earlier.append(c)
    return tokens


def sample_batch(parents, drafts, uniforms):
    """sample_tree for every tree of a batch: parents [B, N+1] int,
    drafts [B, N+1, V] (rows of leaves unused), uniforms [B, N+1].
    Returns (tokens [B, N+1] int64, margins [B, N+1] float64)."""
    parents = np.asarray(parents)
    out = np.zeros(parents.shape, dtype=np.int64)
    marg = np.full(parents.shape, np.inf)
    for b in range(parents.shape[0]):
        m = []
        out[b] = sample_tree(parents[b], np.asarray(drafts[b], dtype=np.float64),
                             [float(x) for x in np.asarray(uniforms[b])], margins=m)
        marg[b] = m
    return out, marg
