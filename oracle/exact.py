"""Exact output laws of Traversal Verification by enumeration.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

``outcome_law`` explores every accept / reject branch of Algorithm 3 on one
fixed draft tree (each test accepts with probability p, rejects with 1 - p;
nodes of rate 0 are removed with certainty) and returns the exact law of
(accepted node, bonus token).  ``z_law`` then averages over the draft trees
of a shape (Definition 1) and extends the output to the fixed length
gamma_max with the target model, giving the sequence Z^{gamma_max} of
Lemma 1 (Appendix A), whose law must equal M_b(.|X_0) for a valid verifier
(Theorem 1).
"""

import itertools
from collections import defaultdict

from workloads.toy_lm import enumerate_draft_trees, node_prefixes

from .traversal import TraversalState

REJECTED = None   # outcome key: the root itself was rejected (root_rate < 1)


def outcome_law(parents, tokens, target_row, draft_row, vocab, root_rate=None,
                allow_zero_draft=False, allow_duplicate_siblings=False):
    """{(accepted node, y): probability}; with ``root_rate`` < 1 the root is
    tested like any node and its rejection yields the key (None, None)."""
    st = TraversalState(parents, tokens, target_row, draft_row, vocab,
                        root_rate=root_rate, allow_zero_draft=allow_zero_draft,
                        allow_duplicate_siblings=allow_duplicate_siblings)
    law = defaultdict(int)

    def explore(state, prob):
        leaf = state.first_leaf()
        p = state.p[leaf]
        if leaf == 0 and root_rate is None:
            p = state.one
        if p > 0:
            w = state.bonus_weights(leaf)
            W = w.sum()
            for y in range(vocab):
                if w[y]:
                    law[(leaf, y)] += prob * p * w[y] / W
        if p < state.one:
            if leaf == 0:
                law[(REJECTED, REJECTED)] += prob * (1 - p)
            else:
                nxt = state.clone()
                nxt.reject(leaf)
                explore(nxt, prob * (1 - p))

    explore(st, st.one)
    return dict(law)


def z_law(parents, mb_table, ms_table, vocab, root_rate=None,
          with_replacement=False, outcome=None):
    """Law of Z^{gamma_max} (Lemma 1) averaged over the draft trees of the
    shape ``parents``: Z = X^tau if tau = gamma_max, else (X^tau, Y, Z_{>tau+1})
    with the tail drawn from the target model.  Keys are token tuples (root
    excluded); the key None collects the mass where the root was rejected.
    ``outcome`` is the verifier's exact outcome law on one tree (default:
    Traversal Verification's ``outcome_law``; the token-level verifier's has
    the same signature)."""
    outcome = outcome_law if outcome is None else outcome
    n = len(parents)
    depth = [0] * n
    for i in range(1, n):
        depth[i] = depth[parents[i]] + 1
    gmax = max(depth)
    law = defaultdict(int)

    def extend(z, q):
        if len(z) == gmax:
            law[z] += q
            return
        row = mb_table[z]
        for t in range(vocab):
            if row[t]:
                extend(z + (t,), q * row[t])

    total = 0
    for tokens, prob in enumerate_draft_trees(parents, ms_table, vocab,
                                              with_replacement=with_replacement):
        total += prob
        pre = node_prefixes(parents, tokens)
        out = outcome(parents, tokens,
                          target_row=lambda i: mb_table[pre[i]].copy(),
                          draft_row=lambda i: ms_table[pre[i]].copy(),
                          vocab=vocab, root_rate=root_rate,
                          allow_zero_draft=with_replacement,
                          allow_duplicate_siblings=with_replacement)
        for (a, y), q in out.items():
            if a is REJECTED:
                law[None] += prob * q
                continue
            z = pre[a]
            if len(z) == gmax:
                law[z] += prob * q
            else:
                extend(z + (y,), prob * q)
    if total != 1 and abs(float(total) - 1.0) > 1e-12:
        raise ValueError("the draft model cannot produce this tree shape "
                         "(a support smaller than a node's branching)")
    return dict(law), gmax


def target_law(mb_table, vocab, length):
    """M_b(z_1..z_L | X_0) for every token sequence of the given length."""
    out = {}
    for z in itertools.product(range(vocab), repeat=length):
        q = 1
        for j in range(length):
            q = q * mb_table[z[:j]][z[j]]
        out[z] = q
    return out
