"""Traversal Verification (Algorithm 3, §3.1) -- literal, materialised, slow.

TEST INFRASTRUCTURE ONLY: imported by tests/, the smoke check and the CPU
legs of bench.py, never by the product path.

Every distribution the algorithm touches is held as a full vector over the
vocabulary and replaced by exactly what Eqs. (1)-(3) of §3.1 prescribe after
each rejection; the rates of the remaining chains are recomputed top-down
after each rejection, as Algorithm 3 states.  Nothing is done in closed form.
The arithmetic is whatever the caller's vectors hold: float64 NumPy arrays
for the parity oracle, NumPy object arrays of ``fractions.Fraction`` for the
exact pins.

Readings taken where the paper leaves a choice (each is listed in the design
notes of the repository):

* Traversal order: the "first" root-to-leaf chain follows the first remaining
  child (children ordered by index) from the root, i.e. a post-order walk
  (Appendix E; the example order X3, X4, X1, X5, X2 of §3.2).
* A node whose rate has reached 0 cannot be accepted any more and is removed
  together with what remains of its subtree (§3.2).  It is removed when the
  first chain reaches it -- exactly when the algorithm would test it and
  reject it with certainty -- so no uniform is drawn for it and the order of
  every other decision is unchanged.  Its removal updates its parent like any
  rejection.
* S = 0 in Eqs. (1)/(3) (a 0/0): for p < 1 the node gets p' = 0 (it will be
  removed as above and its residual is never used); for p = 1 the node keeps
  p' = 1 and its target distribution.  Eq. (2) is applied in both cases.
* The root is never tested: once all its children are gone the root-only
  chain is accepted with tau = 0 (p(X_0) = 1 throughout, since Eq. (3) at
  p = 1 gives S / S = 1).
* A drafted token with M_s(x) = 0 cannot come from Definition 1 and is
  rejected as an invalid tree unless ``allow_zero_draft`` is set (used only
  by the with-replacement negative control), in which case
  min(c / 0, 1) is read as 1 for c > 0 and 0 for c = 0.
* Eq. (2) with 1 - M_s(x_rej) <= 0 (the rejected token held all the draft
  mass left, e.g. the siblings exhausted the support): M_s' is all zero.
"""

import copy

import numpy as np


class InvalidTree(ValueError):
    """The inputs do not form a decoding tree in the sense of Definition 1."""


def _one_like(x):
    return x - x + 1


def _zero_like(x):
    return x - x


def acceptance_rate(p_parent, mb_x, ms_x, allow_zero_draft=False):
    """Sequence-level acceptance rate of a child drafting token x:
    min(p_parent * M_b(x | parent) / M_s(x | parent), 1).

    Used for the initial rates of Algorithm 3 and for the refresh of the
    remaining chains after each rejection (same formula, current
    distributions)."""
    num = p_parent * mb_x
    if ms_x == 0:
        if not allow_zero_draft:
            raise InvalidTree("drafted token has zero draft probability")
        return _one_like(num) if num > 0 else _zero_like(num)
    r = num / ms_x
    one = _one_like(r)
    return r if r < one else one


def residual_mass(p, mb, ms):
    """S = sum_x [p * M_b(x) - M_s(x)]_+ : the normaliser of Eq. (1) and the
    numerator of Eq. (3)."""
    return np.maximum(p * mb - ms, 0).sum()


def residual_target(p, mb, ms, S):
    """Eq. (1): M_b'(x) = [p * M_b(x) - M_s(x)]_+ / S."""
    return np.maximum(p * mb - ms, 0) / S


def draft_without(ms, x_rej):
    """Eq. (2): M_s'(x_rej) = 0 and M_s'(x) = M_s(x) / (1 - M_s(x_rej))
    for every other x."""
    denom = 1 - ms[x_rej]
    if not denom > 0:
        # the rejected token held all the remaining draft mass (the siblings
        # exhausted the support): nothing is left to draft at this node
        return ms * 0
    out = ms / denom
    out[x_rej] = _zero_like(out[x_rej])
    return out


def updated_rate(p, S):
    """Eq. (3): p' = S / (S + 1 - p)."""
    return S / (S + 1 - p)


def validate_tree(parents, tokens, vocab, allow_duplicate_siblings=False):
    """Structural checks of a decoding tree (Definition 1): row 0 is the root,
    every other node's parent precedes it, tokens lie in the vocabulary and
    siblings carry distinct tokens (children drawn without replacement)."""
    n = len(parents)
    if n < 1 or parents[0] != -1:
        raise InvalidTree("row 0 must be the root (parent -1)")
    for i in range(1, n):
        if not 0 <= parents[i] < i:
            raise InvalidTree(f"parent of node {i} must lie in [0, {i})")
        if not 0 <= tokens[i] < vocab:
            raise InvalidTree(f"token of node {i} outside the vocabulary")
    if not allow_duplicate_siblings:
        seen = {}
        for i in range(1, n):
            key = (parents[i], tokens[i])
            if key in seen:
                raise InvalidTree(f"nodes {seen[key]} and {i} are siblings with the same token")
            seen[key] = i


def _condition(p, mb, ms, S):
    """Instrumentation only: relative sensitivity of S to relative
    perturbations of M_b, sum over the positive part of p M_b(x), divided by
    S.  A float computation of S whose M_b values carry a relative error e
    has a relative error of about e times this number."""
    pos = (p * mb - ms) > 0
    if not S > 0:
        # the 0/0 of Eqs. (1)/(3) is resolved exactly (p' = 0 removes the
        # node, p = 1 keeps its row), so no rounding error flows from it
        return 1.0
    return float((p * mb)[pos].sum() / S)


def _cancellation(u, v):
    """Instrumentation only: condition number (|u| + |v|) / |u - v| of u - v."""
    diff = abs(float(u) - float(v))
    tot = abs(float(u)) + abs(float(v))
    return float("inf") if diff == 0 else tot / diff


class TraversalState:
    """Mutable state of Algorithm 3 on one decoding tree.

    ``target_row(i)`` / ``draft_row(i)`` return fresh copies of the original
    M_b(.|X^i) / M_s(.|X^i).  The target rows of all internal nodes and
    their draft rows are materialised up front, as the initialisation of
    Algorithm 3 (rates of all chains) needs them; a leaf's target row is
    fetched only if that leaf is accepted (the bonus token is drawn from it).
    ``root_rate`` (default 1) lets the exact tests run the algorithm on a
    sub-tree whose root has an arbitrary rate, as in Lemma 2.
    """

    def __init__(self, parents, tokens, target_row, draft_row, vocab,
                 root_rate=None, allow_zero_draft=False,
                 allow_duplicate_siblings=False):
        parents = [int(x) for x in parents]
        tokens = [int(x) for x in tokens]
        validate_tree(parents, tokens, vocab, allow_duplicate_siblings)
        n = len(parents)
        self.n = n
        self.parents = parents
        self.tokens = tokens
        self.children = [[] for _ in range(n)]
        for i in range(1, n):
            self.children[parents[i]].append(i)
        self.depth = [0] * n
        for i in range(1, n):
            self.depth[i] = self.depth[parents[i]] + 1
        self.alive = [True] * n
        self.allow_zero_draft = allow_zero_draft
        self._target_row = target_row
        self.mb = {}
        self.ms = {}
        for i in range(n):
            if self.children[i]:
                self.mb[i] = target_row(i)
                self.ms[i] = draft_row(i)
        # instrumentation: S-computations per node, degenerate S == 0 events,
        # nodes removed with rate 0, and the bonus row fetched for a leaf
        self.passes = [0] * n
        self.kappa = []         # condition number of each S (instrumentation)
        self.kappa_S = []       # the S each kappa entry belongs to (instrumentation)
        self.degenerate = 0
        self.pruned = []
        self.leaf_rows_read = set()
        # initial acceptance rates of every node of every chain, top-down
        # (parents precede children in index order)
        if n > 1:
            one = _one_like(self.mb[0][0])
        else:
            one = 1.0
        self.one = one
        self.p = [None] * n
        self.p[0] = one if root_rate is None else root_rate * one
        for i in range(1, n):
            self.p[i] = self._rate_of(i)

    def clone(self):
        return copy.deepcopy(self)

    def _rate_of(self, i):
        par = self.parents[i]
        x = self.tokens[i]
        return acceptance_rate(self.p[par], self.mb[par][x], self.ms[par][x],
                               self.allow_zero_draft)

    def _subtree(self, i):
        out = [i]
        k = 0
        while k < len(out):
            out.extend(self.children[out[k]])
            k += 1
        return out

    def _is_descendant(self, d, i):
        while d > i:
            d = self.parents[d]
        return d == i

    def remaining_children(self, i):
        return [c for c in self.children[i] if self.alive[c]]

    def first_leaf(self):
        """Last node of the root-to-first-leaf chain of the remaining tree.

        Nodes of rate 0 met on the way are removed with their subtree (and
        their parent updated) before the chain is re-selected."""
        while True:
            node = 0
            while True:
                kids = self.remaining_children(node)
                if not kids:
                    return node
                c = kids[0]
                if self.p[c] == 0:
                    self.pruned.append(c)
                    self.reject(c)
                    break
                node = c

    def reject(self, c):
        """Delete node c (and anything left below it), then update its parent
        by Eqs. (1), (2) and (3) and refresh the rates of the parent's
        remaining descendants."""
        if c == 0:
            raise ValueError("the root is never deleted")
        for d in self._subtree(c):
            self.alive[d] = False
        i = self.parents[c]
        p = self.p[i]
        mb, ms = self.mb[i], self.ms[i]
        S = residual_mass(p, mb, ms)
        self.passes[i] += 1
        self.kappa.append(_condition(p, mb, ms, S))
        self.kappa_S.append(float(S))
        if S > 0:
            new_mb = residual_target(p, mb, ms, S)
            new_p = updated_rate(p, S)
            # instrumentation: cancellation in the residual of every remaining
            # child's token, on top of that of S
            for d in self.children[i]:
                if self.alive[d]:
                    x = self.tokens[d]
                    self.kappa.append(self.kappa[-1] + _cancellation(p * mb[x], ms[x]))
                    self.kappa_S.append(float(S))
        else:
            self.degenerate += 1
            new_mb = mb
            new_p = self.one if p == self.one else _zero_like(self.one)
        new_ms = draft_without(ms, self.tokens[c])
        self.mb[i], self.ms[i], self.p[i] = new_mb, new_ms, new_p
        for d in range(i + 1, self.n):
            if self.alive[d] and self._is_descendant(d, i):
                self.p[d] = self._rate_of(d)

    def bonus_weights(self, a):
        """Current M_b(.|X^a) of the accepted node: the residual left by the
        rejections at a if a had children, else a's original target row."""
        if a in self.mb:
            return self.mb[a]
        self.leaf_rows_read.add(a)
        return self._target_row(a)

    def path(self, a):
        out = []
        while a != 0:
            out.append(a)
            a = self.parents[a]
        return out[::-1]
