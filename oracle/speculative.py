"""Token-level verifiers the paper builds on, written from their own
definitions so that Traversal Verification can be pinned against them.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

* ``single_token_law``  -- Algorithm 1 (single-token verification, §2.1).
* ``rrs_law``           -- Algorithm 2 (Recursive Rejection Sampling, §2.2),
  with or without replacement.

Both return the exact output law as a dict {(accepted candidate or None, y):
probability} for fixed inputs, computed with whatever arithmetic the vectors
carry (float64 or Fraction object arrays).
"""

import numpy as np


def _normalise(v):
    tot = v.sum()
    return v / tot if tot else v * 0


def single_token_law(mb_root, ms_root, x, mb_child):
    """Algorithm 1: the draft token x (drawn from M_s(.|X0)) is accepted with
    probability min(1, M_b(x)/M_s(x)); then Y ~ M_b(.|X0, x).  On rejection
    Y ~ norm([M_b - M_s]_+) at the prefix."""
    ratio = mb_root[x] / ms_root[x]
    acc = ratio if ratio < 1 else ratio - ratio + 1
    law = {}
    for y, w in enumerate(mb_child):
        if w:
            law[(x, y)] = law.get((x, y), 0) + acc * w
    rej = 1 - acc
    if rej:
        resid = _normalise(np.maximum(mb_root - ms_root, 0))
        for y, w in enumerate(resid):
            if w:
                law[(None, y)] = law.get((None, y), 0) + rej * w
    return law


def rrs_law(mb_root, ms_root, candidates, mb_children, without_replacement=True):
    """Algorithm 2: candidates X_1..X_k are tried in order; X_i is accepted
    with probability min(1, M_b'(X_i)/M_s'(X_i)) and then Y ~ M_b(.|X0, X_i);
    each rejection sets M_b' <- norm([M_b' - M_s']_+) and, without
    replacement, M_s' <- norm(M_s' with M_s'(X_i) = 0).  If every candidate
    is rejected, Y ~ M_b'.  ``mb_children[i]`` is M_b(.|X0, X_i)."""
    law = {}
    mb = mb_root.copy()
    ms = ms_root.copy()
    reach = mb[0] - mb[0] + 1          # probability of reaching candidate i
    for i, x in enumerate(candidates):
        if ms[x] == 0:
            acc = reach - reach + (1 if mb[x] > 0 else 0)
        else:
            r = mb[x] / ms[x]
            acc = r if r < 1 else r - r + 1
        for y, w in enumerate(mb_children[i]):
            if w:
                law[(i, y)] = law.get((i, y), 0) + reach * acc * w
        reach = reach * (1 - acc)
        if not reach:
            return law
        mb = _normalise(np.maximum(mb - ms, 0))
        if without_replacement:
            ms = ms.copy()
            ms[x] = ms[x] - ms[x]
            ms = _normalise(ms)
    for y, w in enumerate(mb):
        if w:
            law[(None, y)] = law.get((None, y), 0) + reach * w
    return law
