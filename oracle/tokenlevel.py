"""Token-level tree verification -- the top-down verifier that Traversal
Verification is compared with (§2.2, the verification order described for
the two-layer tree of Fig. 2; "Tok.V" in §4) -- literal, materialised, slow.

TEST INFRASTRUCTURE ONLY: imported by tests/, the smoke check and the CPU
legs of bench.py, never by the product path.

At the current node (the root first) its children are the candidates of one
run of Recursive Rejection Sampling without replacement (Algorithm 2, §2.2):
child X_i is accepted with probability min(1, M_b'(x_i) / M_s'(x_i)) under
the node's current pair (M_b', M_s'); a rejection sets
M_b' <- norm([M_b' - M_s']_+) and removes x_i from M_s' (renormalising the
rest).  An accepted child becomes the current node with its own, untouched
distributions, so a rejected child's subtree is never looked at.  Once the
current node has no candidate left -- it is a leaf, or all its children were
rejected -- the bonus token is drawn from its current M_b'.

Every distribution is a full vector over the vocabulary; the arithmetic is
whatever the caller's vectors hold (float64 arrays for the parity oracle,
object arrays of ``fractions.Fraction`` for the exact pins).

Readings (the same as the traversal oracle's where they apply):

* one pre-drawn uniform per node (u[i] tests node i, u[N+1] draws Y) and the
  strict test u < p;
* siblings are drafted without replacement, in child order; a drafted token
  with M_s'(x) = 0 cannot come from Definition 1 and makes the tree invalid
  (unless ``allow_zero_draft``, used by the with-replacement control);
* a child of rate 0 is tested and rejected like any other (it has a uniform);
* a rejection whose residual vanishes (sum_x [M_b' - M_s']_+ = 0, which needs
  M_b' = M_s' and hence a rate of 1, so only rounding reaches it) keeps M_b'
  and still removes the token from M_s'; it is counted as degenerate.
"""

import copy
from collections import defaultdict

import numpy as np

from .traversal import (InvalidTree, _cancellation, _condition, _one_like, acceptance_rate,
                        draft_without, residual_mass, residual_target, validate_tree)
from .verify import inverse_cdf, softmax_f64, verify_batch


class TokenLevelState:
    """Mutable state of the top-down verifier on one decoding tree.

    ``target_row(i)`` / ``draft_row(i)`` return fresh copies of the original
    M_b(.|X^i) / M_s(.|X^i); a row is fetched only when the walk reaches its
    node (the rows of rejected subtrees are never read)."""

    def __init__(self, parents, tokens, target_row, draft_row, vocab,
                 allow_zero_draft=False, allow_duplicate_siblings=False):
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
        self.allow_zero_draft = allow_zero_draft
        self._target_row = target_row
        self._draft_row = draft_row
        # instrumentation: S-computations per node, rows whose target
        # distribution the walk needed, condition numbers of each S
        self.passes = [0] * n
        self.kappa = []
        self.degenerate = 0
        self.rows_read = []
        self._enter(0)
        self.one = _one_like(self.mb[0]) if len(self.mb) else 1.0

    def clone(self):
        return copy.deepcopy(self)

    def _enter(self, i):
        """Make node i the current node, with its original distributions."""
        self.node = i
        self.next = 0
        self.mb = self._target_row(i)
        self.rows_read.append(i)
        self.ms = self._draft_row(i) if self.children[i] else None

    def candidate(self):
        """Next child of the current node to test, or None (no candidate left)."""
        kids = self.children[self.node]
        return kids[self.next] if self.next < len(kids) else None

    def rate(self, c):
        """min(1, M_b'(x_c) / M_s'(x_c)) under the current node's pair."""
        x = self.tokens[c]
        return acceptance_rate(self.one, self.mb[x], self.ms[x], self.allow_zero_draft)

    def accept(self, c):
        self._enter(c)

    def reject(self, c):
        """Residual update of Algorithm 2 (without replacement) at the current node."""
        S = residual_mass(self.one, self.mb, self.ms)
        self.passes[self.node] += 1
        self.kappa.append(_condition(self.one, self.mb, self.ms, S))
        if S > 0:
            # instrumentation: cancellation in the residual of every sibling
            # still to be tested, on top of that of S
            for d in self.children[self.node][self.next + 1:]:
                x = self.tokens[d]
                self.kappa.append(self.kappa[-1] + _cancellation(self.mb[x], self.ms[x]))
            self.mb = residual_target(self.one, self.mb, self.ms, S)
        else:
            self.degenerate += 1
        self.ms = draft_without(self.ms, self.tokens[c])
        self.next += 1

    def bonus_weights(self):
        """Current M_b' of the node the walk stopped at."""
        return self.mb

    def path(self):
        out = []
        a = self.node
        while a != 0:
            out.append(a)
            a = self.parents[a]
        return out[::-1]


def outcome_law(parents, tokens, target_row, draft_row, vocab, root_rate=None,
                allow_zero_draft=False, allow_duplicate_siblings=False):
    """Exact law {(node the walk stopped at, y): probability} of the
    top-down verifier on one fixed draft tree, exploring every accept /
    reject branch (``root_rate`` is not meaningful here and must be None)."""
    if root_rate is not None:
        raise ValueError("the token-level verifier never tests the root")
    st = TokenLevelState(parents, tokens, target_row, draft_row, vocab,
                         allow_zero_draft=allow_zero_draft,
                         allow_duplicate_siblings=allow_duplicate_siblings)
    law = defaultdict(int)

    def explore(state, prob):
        c = state.candidate()
        if c is None:
            w = state.bonus_weights()
            W = w.sum()
            for y in range(vocab):
                if w[y]:
                    law[(state.node, y)] += prob * w[y] / W
            return
        p = state.rate(c)
        if p > 0:
            nxt = state.clone()
            nxt.accept(c)
            explore(nxt, prob * p)
        if p < state.one:
            nxt = state.clone()
            nxt.reject(c)
            explore(nxt, prob * (1 - p))

    explore(st, st.one)
    return dict(law)


def verify_tree(parents, tokens, logits, draft_probs, temperature, uniforms, keep_cdf=False):
    """Token-level verification of one tree; same inputs and result fields
    as the traversal oracle's ``verify_tree`` (``pruned`` is always empty:
    a rejected child's subtree is simply never reached)."""
    parents = np.asarray(parents).astype(np.int64)
    tokens = np.asarray(tokens).astype(np.int64)
    n = len(parents)
    V = logits.shape[1]
    T = float(np.float32(temperature))
    if not T > 0:
        raise ValueError("temperature must be > 0 (the method needs sampling)")
    u = np.asarray(uniforms, dtype=np.float64)
    st = TokenLevelState(parents, tokens,
                         target_row=lambda i: softmax_f64(logits[i], T),
                         draft_row=lambda i: np.asarray(draft_probs[i], dtype=np.float64),
                         vocab=V)
    node_p = np.full(n, np.nan)
    tests = []
    kappa_at_test = []
    while True:
        c = st.candidate()
        if c is None:
            break
        p = float(st.rate(c))
        node_p[c] = p
        tests.append((c, float(u[c]), p))
        kappa_at_test.append(max(st.kappa, default=1.0))
        if u[c] < p:
            st.accept(c)
        else:
            st.reject(c)
    accepted = st.node
    w = st.bonus_weights()
    y, y_margin, W = inverse_cdf(w, u[n])
    cdf = np.cumsum(np.asarray(w, dtype=np.float64)) if keep_cdf else None
    path = st.path()
    internal = [i for i in range(n) if st.children[i]]
    return {
        "path": path,
        "tau": len(path),
        "bonus": y,
        "accepted": accepted,
        "node_p": node_p,
        "tests": tests,
        "kappa_at_test": kappa_at_test,
        "test_margin": min((abs(uu - pp) for _, uu, pp in tests), default=np.inf),
        "bonus_margin": y_margin,
        "bonus_total": W,
        "passes": list(st.passes),
        "n_passes": int(sum(st.passes)),
        "rejected_at": [i for i in range(n) if st.passes[i] > 0],
        "internal": internal,
        "rows_read": list(st.rows_read),
        "leaf_row_read": not st.children[accepted],
        "pruned": [],
        "degenerate": st.degenerate,
        "bonus_u": float(u[n]),
        "bonus_cdf": cdf,
    }


def verify_batch_token_level(parents, tokens, logits, draft_probs, temperature, uniforms,
                             trees=None, keep_cdf=False):
    """Batch driver (same arrays and marking of invalid trees as the traversal
    oracle's ``verify_batch``)."""
    return verify_batch(parents, tokens, logits, draft_probs, temperature, uniforms,
                        trees=trees, keep_cdf=keep_cdf, tree_fn=verify_tree)


__all__ = ["InvalidTree", "TokenLevelState", "outcome_law", "verify_tree",
           "verify_batch_token_level"]
