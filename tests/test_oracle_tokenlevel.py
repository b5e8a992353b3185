"""Pins of the token-level tree verifier of the oracle (oracle/tokenlevel.py).

Checked against what the paper and the mathematics fix, not against itself:
the token-level value the paper prints for its worked example (§3.2) and the
rest of that law derived by hand from §2.2's verification order; the
algorithms it is built from (Algorithm 1 for one node, Algorithm 2 for one
layer, written separately in oracle/speculative.py); losslessness by exact
enumeration; and Theorem 2's statement that Traversal Verification is at
least as long on a chain.  Planted mistakes must fail the enumeration.
"""

import json
import os
from fractions import Fraction as F

import numpy as np
import pytest

import oracle.tokenlevel as tok
from oracle.exact import outcome_law as traversal_law
from oracle.exact import target_law, z_law
from oracle.speculative import rrs_law, single_token_law
from oracle.traversal import InvalidTree
from workloads.toy_lm import enumerate_draft_trees, node_prefixes, rational_table

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example.json")


def frac_vec(xs):
    return np.array([F(x) for x in xs], dtype=object)


@pytest.fixture(scope="module")
def example():
    with open(GOLDEN) as f:
        return json.load(f)


def _example_tree(example):
    t = example["traversal"]
    idx = {"a": 0, "b": 1, "c": 2}
    return t["parents"], [0] + [idx[x] for x in t["tokens"][1:]]


def _accepted(law):
    acc = {}
    for (a, _), q in law.items():
        acc[a] = acc.get(a, 0) + q
    return acc


# ------------------------------------------------------ worked example ----

def test_example_tree_token_level_law(example):
    """§3.2's tree with M_b = [.3,.4,.3], M_s = [.6,.3,.1] at every context,
    verified top-down (§2.2): X1 = a is accepted w.p. min(.3/.6, 1) = 1/2 and
    then X3 = b w.p. min(.4/.3, 1) = 1, so P(X1 X3) = 1/2 -- the value the
    paper prints for token-level verification.  If X1 is rejected the root's
    pair becomes [0,1/3,2/3] / [0,3/4,1/4] (the RRSw example), X2 = c is
    accepted w.p. 1, then X5 = a w.p. 1/2; rejecting X5 leaves X2 with the
    residual [0,1/3,2/3] for the bonus token."""
    mb = frac_vec(example["M_b"])
    ms = frac_vec(example["M_s"])
    parents, toks = _example_tree(example)
    law = tok.outcome_law(parents, toks, lambda i: mb.copy(), lambda i: ms.copy(), 3)
    acc = _accepted(law)
    assert acc[3] == F(str(example["traversal"]["printed"]["accept_X1X3_token_level"]))
    assert acc == {3: F(1, 2), 5: F(1, 4), 2: F(1, 4)}
    assert law[(2, 1)] / acc[2] == F(1, 3) and law[(2, 2)] / acc[2] == F(2, 3)
    assert (2, 0) not in law
    # the bonus after an accepted leaf comes from that leaf's own row
    for leaf in (3, 5):
        assert [law[(leaf, y)] / acc[leaf] for y in range(3)] == list(mb)
    # Traversal Verification on the same tree: E[tau] = 64/33 > 7/4
    tv = _accepted(traversal_law(parents, toks, lambda i: mb.copy(), lambda i: ms.copy(), 3))
    depth = {0: 0, 1: 1, 2: 1, 3: 2, 4: 2, 5: 2}
    e_tv = sum(q * depth[a] for a, q in tv.items())
    e_tok = sum(q * depth[a] for a, q in acc.items())
    assert e_tok == F(7, 4) and e_tv == F(64, 33)


# ------------------------------------------- reductions to Alg. 1 / 2 -----

@pytest.mark.parametrize("seed", range(6))
def test_single_node_tree_is_algorithm1(seed):
    V = 4
    t = rational_table(V, 1, seed, zero_prob=0.2)
    s = rational_table(V, 1, seed + 50, zero_prob=0.2)
    for x in range(V):
        if s[()][x] == 0:
            continue
        rows_b = {0: t[()], 1: t[(x,)]}
        law = tok.outcome_law([-1, 0], [0, x], lambda i: rows_b[i].copy(),
                              lambda i: s[()].copy(), V)
        ref = single_token_law(t[()], s[()], x, t[(x,)])
        got = {((x if a == 1 else None), y): q for (a, y), q in law.items()}
        assert got == {k: v for k, v in ref.items() if v}


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("k", [2, 3])
def test_depth1_tree_is_rrs_without_replacement(seed, k):
    V = 4
    t = rational_table(V, 1, seed, zero_prob=0.15)
    s = rational_table(V, 1, seed + 70, zero_prob=0.15, min_support=k)
    parents = [-1] + [0] * k
    for tokens, _ in enumerate_draft_trees(parents, s, V):
        cand = tokens[1:]
        rows_b = [t[()]] + [t[(c,)] for c in cand]
        law = tok.outcome_law(parents, tokens, lambda i: rows_b[i].copy(),
                              lambda i: s[()].copy(), V)
        ref = rrs_law(t[()], s[()], cand, [t[(c,)] for c in cand])
        got = {((a - 1) if a != 0 else None, y): q for (a, y), q in law.items()}
        assert got == {kk: v for kk, v in ref.items() if v}


# ------------------------------------------------------ losslessness ------

SHAPES = [
    ([-1, 0, 0, 1, 1, 2], 3),
    ([-1, 0, 1, 2], 4),
    ([-1, 0, 0, 1, 1, 2, 2], 4),
    ([-1, 0, 0, 0, 1, 1, 2, 4], 3),
    ([-1, 0, 1, 1, 2, 3], 3),
]


def _lossless(shape, V, seed, zero_prob=0.0, **kw):
    branching = max(shape[1:].count(i) for i in range(len(shape)))
    t = rational_table(V, 3, seed, zero_prob=zero_prob)
    s = rational_table(V, 3, seed + 1000, zero_prob=zero_prob, min_support=branching)
    zl, g = z_law(shape, t, s, V, outcome=tok.outcome_law, **kw)
    tl = target_law(t, V, g)
    return all(zl.get(z, 0) == q for z, q in tl.items()) and set(zl) <= set(tl)


@pytest.mark.parametrize("shape,V", SHAPES)
@pytest.mark.parametrize("seed", [1, 2])
def test_lossless_exact(shape, V, seed):
    """Z^{gamma_max} of the token-level verifier has the target law exactly."""
    assert _lossless(shape, V, seed)


@pytest.mark.parametrize("seed", [3, 4])
def test_lossless_exact_with_zero_probabilities(seed):
    assert _lossless([-1, 0, 0, 1, 1, 2, 2], 3, seed, zero_prob=0.3)
    assert _lossless([-1, 0, 0, 0, 1, 2], 4, seed, zero_prob=0.3)


def test_negative_control_with_replacement():
    results = [_lossless([-1, 0, 0, 1, 1, 2, 2], 3, seed, with_replacement=True)
               for seed in (3, 5, 7)]
    assert not all(results)


MUTATIONS = {
    "draft row not updated": ("draft_without", lambda ms, x: ms.copy()),
    "residual not renormalised": ("residual_target",
                                  lambda p, mb, ms, S: np.maximum(p * mb - ms, 0)),
}


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_planted_mistakes_fail(monkeypatch, name):
    attr, fn = MUTATIONS[name]
    monkeypatch.setattr(tok, attr, fn)
    ok = True
    for shape, V in SHAPES[:3]:
        try:
            ok = ok and _lossless(shape, V, 1)
        except (ZeroDivisionError, InvalidTree, ValueError):
            ok = False
    assert not ok


# ------------------------------------------------------ Theorem 2 ---------

@pytest.mark.parametrize("seed", [5, 6, 7, 8])
def test_traversal_at_least_as_long_on_chains(seed):
    """Theorem 2: on a chain, Traversal Verification's E[tau] is at least the
    token-level verifier's, whose E[tau] is sum_l prod_{j<=l} min(r_j, 1)."""
    V = 3
    shape = [-1, 0, 1, 2]
    t = rational_table(V, 3, seed)
    s = rational_table(V, 3, seed + 1000)
    e_tv = e_tok = e_closed = 0
    for tokens, prob in enumerate_draft_trees(shape, s, V):
        pre = node_prefixes(shape, tokens)
        rows_b = lambda i: t[pre[i]].copy()
        rows_s = lambda i: s[pre[i]].copy()
        for (a, _), q in traversal_law(shape, tokens, rows_b, rows_s, V).items():
            e_tv += prob * q * len(pre[a])
        for (a, _), q in tok.outcome_law(shape, tokens, rows_b, rows_s, V).items():
            e_tok += prob * q * len(pre[a])
        acc = F(1)
        for l in range(1, len(shape)):
            acc = acc * min(t[pre[l - 1]][tokens[l]] / s[pre[l - 1]][tokens[l]], F(1))
            e_closed += prob * acc
    assert e_tok == e_closed
    assert e_tv >= e_tok


# ------------------------------------------------------ float driver ------

@pytest.mark.parametrize("seed", range(8))
def test_float_driver_follows_the_exact_walk(seed):
    """The float64 driver takes the same decisions and rates as the exact
    state machine fed the same uniforms."""
    rng = np.random.default_rng(seed)
    V, parents = 5, [-1, 0, 0, 0, 1, 1, 2, 4]
    n = len(parents)
    logits = rng.normal(size=(n, V)) * 2
    drafts = rng.dirichlet(np.ones(V), size=n)
    tokens = [0]
    for i in range(1, n):
        sib = [tokens[j] for j in range(1, i) if parents[j] == parents[i]]
        free = [x for x in range(V) if x not in sib]
        tokens.append(int(rng.choice(free)))
    u = rng.random(n + 1)
    u[0] = 0.0
    r = tok.verify_tree(parents, tokens, logits, drafts, 1.0, u)
    mb = lambda i: np.array([F(float(x)) for x in tok.softmax_f64(logits[i], 1.0)], dtype=object)
    ms = lambda i: np.array([F(float(x)) for x in drafts[i]], dtype=object)
    st = tok.TokenLevelState(parents, tokens, mb, ms, V)
    while True:
        c = st.candidate()
        if c is None:
            break
        p = st.rate(c)
        assert abs(float(p) - r["node_p"][c]) < 1e-12
        if F(float(u[c])) < p:
            st.accept(c)
        else:
            st.reject(c)
    assert st.path() == r["path"] and r["tau"] == len(r["path"])
    assert [c for c, _, _ in r["tests"]] == [c for c in range(1, n) if not np.isnan(r["node_p"][c])]


def test_invalid_trees_are_marked():
    V, n = 4, 3
    logits = np.zeros((1, n, V))
    drafts = np.full((1, n, V), 0.25)
    parents = np.array([[-1, 0, 0]])
    tokens = np.array([[0, 2, 2]])       # duplicate siblings
    u = np.zeros((1, n + 1))
    _, tau, bonus, det = tok.verify_batch_token_level(parents, tokens, logits, drafts, 1.0, u)
    assert tau[0] == -1 and bonus[0] == -1 and "invalid" in det[0]
