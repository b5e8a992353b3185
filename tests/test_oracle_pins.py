"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: values the
paper prints for its worked examples (tests/golden/worked_example.json), the
token-level algorithms it reduces to (Algorithms 1 and 2, written separately
in oracle/speculative.py), and the exact laws its theorems state (Lemma 1,
Lemma 2, Theorems 1 and 2), checked by exhaustive enumeration in exact
rational arithmetic.  Planted mistakes must make the same checks fail.
"""

import json
import os
from fractions import Fraction as F

import numpy as np
import pytest

import oracle.traversal as tv
from oracle.exact import outcome_law, target_law, z_law
from oracle.speculative import rrs_law, single_token_law
from oracle.traversal import InvalidTree, TraversalState
from workloads.toy_lm import (enumerate_draft_trees, node_prefixes,
                              rational_table)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example.json")


def frac_vec(xs):
    return np.array([F(x) for x in xs], dtype=object)


@pytest.fixture(scope="module")
def example():
    with open(GOLDEN) as f:
        return json.load(f)


def ex_rows(example):
    mb = frac_vec(example["M_b"])
    ms = frac_vec(example["M_s"])
    return mb, ms


def ex_tree(example):
    t = example["traversal"]
    idx = {"a": 0, "b": 1, "c": 2}
    toks = [0] + [idx[x] for x in t["tokens"][1:]]
    return t["parents"], toks


# ---------------------------------------------------------------- P1 ------

def test_worked_example_trajectory(example):
    """§3.2: every intermediate value of the traversal of the example tree."""
    mb, ms = ex_rows(example)
    parents, toks = ex_tree(example)
    ex = {k: (F(v) if isinstance(v, str) else v)
          for k, v in example["traversal"]["exact"].items()}
    st = TraversalState(parents, toks, lambda i: mb.copy(), lambda i: ms.copy(), 3)
    assert st.p[1] == ex["p_X1"]
    assert st.p[3] == ex["accept_X1X3"]
    # the first chain ends in X3
    assert st.first_leaf() == 3
    assert tv.residual_mass(st.p[1], st.mb[1], st.ms[1]) == ex["S_after_X3"]
    st.reject(3)
    assert st.p[1] == ex["p_prime_X1"]
    assert st.first_leaf() == 4
    assert st.p[4] == ex["accept_X1X4"]
    assert tv.residual_mass(st.p[1], st.mb[1], st.ms[1]) == ex["S_after_X4"]
    st.reject(4)
    assert st.p[1] == ex["p_X1_after_X4"]
    # X1 (rate 0) is removed when the chain reaches it; X5 is next
    assert st.first_leaf() == 5
    assert st.pruned == [1]
    assert list(st.mb[0]) == [F(x) for x in ex["root_M_b_after_X1"]]
    assert list(st.ms[0]) == [F(x) for x in ex["root_M_s_after_X1"]]
    assert st.p[0] == 1
    assert st.p[2] == ex["p_X2"]
    assert st.p[5] == ex["p_X5"]
    st.reject(5)
    assert st.first_leaf() == 2


def test_worked_example_printed_values(example):
    """The decimals §3.2 prints, within their printed rounding; 0.637 is the
    paper's product of the rounded p' = 0.091 with the ratio 7 (reading in
    the fixture), the exact value being 7/11."""
    pr = example["traversal"]["printed"]
    ex = example["traversal"]["exact"]
    assert abs(float(F(ex["accept_X1X3"])) - pr["accept_X1X3"]) < 5e-4
    assert abs(float(F(ex["p_prime_X1"])) - pr["p_prime_X1"]) < 5e-4
    assert abs(7 * pr["p_prime_X1"] - pr["accept_X1X4"]) < 1e-9
    assert abs(float(F(ex["accept_X1X4"])) - pr["accept_X1X4"]) < 1.5e-3
    # token-level acceptance of the same chain, min(r1,1)*min(r3,1)
    assert F(1, 2) * 1 == F(str(pr["accept_X1X3_token_level"]))


def test_worked_example_order_and_law(example):
    """Traversal order X3, X4, X1, X5, X2 (§3.2) and the resulting law of the
    accepted node, built from the printed conditional acceptance rates."""
    mb, ms = ex_rows(example)
    parents, toks = ex_tree(example)
    law = outcome_law(parents, toks, lambda i: mb.copy(), lambda i: ms.copy(), 3)
    acc = {}
    for (a, _), q in law.items():
        acc[a] = acc.get(a, 0) + q
    p3, p4, p5 = F(2, 3), F(7, 11), F(1, 2)
    assert acc[3] == p3
    assert acc[4] == (1 - p3) * p4
    assert acc[5] == (1 - p3) * (1 - p4) * p5
    assert acc[2] == (1 - p3) * (1 - p4) * (1 - p5)
    assert 1 not in acc            # X1 reached rate 0
    assert sum(acc.values()) == 1
    # Y after X2 alone is drawn from the residual at X2: [0, 1/3, 2/3]
    assert (2, 0) not in law
    assert law[(2, 1)] / acc[2] == F(1, 3) and law[(2, 2)] / acc[2] == F(2, 3)
    # visiting order: record the leaves in the order they are tested
    st = TraversalState(parents, toks, lambda i: mb.copy(), lambda i: ms.copy(), 3)
    order = []
    while True:
        leaf = st.first_leaf()
        if leaf == 0:
            break
        order.append(leaf)
        st.reject(leaf)
    seen = order[:2] + st.pruned[:1] + order[2:]
    assert seen == example["traversal"]["order"]


def test_table1_single_token(example):
    """Table 1 (§2.1): a accepted w.p. 1/2, output law equals M_b, residual
    [0, .1, .2] unnormalised."""
    mb, ms = ex_rows(example)
    t1 = example["table1"]
    law = single_token_law(mb, ms, 0, mb)
    assert law[(0, 0)] + law[(0, 1)] + law[(0, 2)] == F(t1["accept_prob_a"])
    assert list(np.maximum(mb - ms, 0)) == [F(x) for x in t1["residual_unnormalised"]]
    # averaged over x ~ M_s the first output token has law M_b
    first = [0, 0, 0]
    for x in range(3):
        lx = single_token_law(mb, ms, x, mb)
        for (a, y), q in lx.items():
            first[x if a is not None else y] += ms[x] * q
    assert first == [F(v) for v in t1["prob_output"].values()]


def test_rrsw_example(example):
    """§2.2: after rejecting a, M_b' = [0,1/3,2/3], M_s' = [0,3/4,1/4], and b
    is then accepted w.p. 4/9 -- reproduced by a depth-1 traversal."""
    mb, ms = ex_rows(example)
    r = example["rrsw"]
    st = TraversalState([-1, 0, 0], [0, 0, 1], lambda i: mb.copy(), lambda i: ms.copy(), 3)
    assert st.first_leaf() == 1
    st.reject(1)
    assert list(st.mb[0]) == [F(x) for x in r["M_b_prime"]]
    assert list(st.ms[0]) == [F(x) for x in r["M_s_prime"]]
    assert st.p[2] == F(r["accept_prob_b"])


# ----------------------------------------------------- P2 / P3 ------------

@pytest.mark.parametrize("seed", range(6))
def test_single_node_tree_is_algorithm1(seed):
    """A one-node tree reduces to single-token verification (Algorithm 1)."""
    V = 4
    t = rational_table(V, 1, seed, zero_prob=0.2)
    s = rational_table(V, 1, seed + 50, zero_prob=0.2)
    for x in range(V):
        if s[()][x] == 0:
            continue
        rows_b = {0: t[()], 1: t[(x,)]}
        law = outcome_law([-1, 0], [0, x], lambda i: rows_b[i].copy(),
                          lambda i: s[()].copy(), V)
        ref = single_token_law(t[()], s[()], x, t[(x,)])
        got = {((x if a == 1 else None), y): q for (a, y), q in law.items()}
        assert got == {k: v for k, v in ref.items() if v}


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("k", [2, 3])
def test_depth1_tree_is_rrsw(seed, k):
    """A depth-1 tree with k children reduces to RRS without replacement
    (Algorithm 2), candidate by candidate."""
    V = 4
    t = rational_table(V, 1, seed, zero_prob=0.15)
    s = rational_table(V, 1, seed + 70, zero_prob=0.15, min_support=k)
    parents = [-1] + [0] * k
    for tokens, _ in enumerate_draft_trees(parents, s, V):
        cand = tokens[1:]
        rows_b = [t[()]] + [t[(c,)] for c in cand]
        law = outcome_law(parents, tokens, lambda i: rows_b[i].copy(),
                          lambda i: s[()].copy(), V)
        ref = rrs_law(t[()], s[()], cand, [t[(c,)] for c in cand])
        got = {((a - 1) if a != 0 else None, y): q for (a, y), q in law.items()}
        assert got == {kk: v for kk, v in ref.items() if v}


# ------------------------------------------------------------ P4 ----------

SHAPES = [
    ([-1, 0, 0, 1, 1, 2], 3),            # the paper's example shape
    ([-1, 0, 1, 2], 4),                  # chain of 3
    ([-1, 0, 0, 1, 1, 2, 2], 4),         # binary depth 2
    ([-1, 0, 0, 0, 1, 1, 2, 4], 3),      # mixed depth 3
    ([-1, 0, 1, 1, 2, 3], 3),            # deep first chain with a side branch
]


def _lossless(shape, V, seed, zero_prob=0.0, **kw):
    branching = max(shape[1:].count(i) for i in range(len(shape)))
    t = rational_table(V, 3, seed, zero_prob=zero_prob)
    s = rational_table(V, 3, seed + 1000, zero_prob=zero_prob, min_support=branching)
    zl, g = z_law(shape, t, s, V, **kw)
    tl = target_law(t, V, g)
    return all(zl.get(z, 0) == q for z, q in tl.items()) and set(zl) <= set(tl)


@pytest.mark.parametrize("shape,V", SHAPES)
@pytest.mark.parametrize("seed", [1, 2])
def test_lossless_exact(shape, V, seed):
    """Theorem 1 via Lemma 1: the law of Z^{gamma_max} equals the target
    model's law exactly (rational arithmetic, every draft tree and every
    accept / reject branch enumerated)."""
    assert _lossless(shape, V, seed)


@pytest.mark.parametrize("seed", [3, 4])
def test_lossless_exact_with_zero_probabilities(seed):
    """Same with distributions that put zero mass on some tokens, which makes
    exact S = 0 and rate-0 removals occur."""
    assert _lossless([-1, 0, 0, 1, 1, 2, 2], 3, seed, zero_prob=0.3)
    assert _lossless([-1, 0, 0, 0, 1, 2], 4, seed, zero_prob=0.3)


def test_negative_control_with_replacement():
    """Drafting siblings with replacement violates the premise of Eq. (2);
    the output law then differs from the target law (so the enumeration has
    the power to see a wrong draft model)."""
    results = [_lossless([-1, 0, 0, 1, 1, 2, 2], 3, seed, with_replacement=True)
               for seed in (3, 5, 7)]
    assert not all(results)


MUTATIONS = {
    "e3 without 1-p": ("updated_rate", lambda p, S: S / (S + 1)),
    "e1 without p": ("residual_target",
                     lambda p, mb, ms, S: np.maximum(mb - ms, 0) / np.maximum(mb - ms, 0).sum()),
    "e2 skipped": ("draft_without", lambda ms, x: ms.copy()),
    "token-level rate": ("acceptance_rate",
                         lambda p, mb, ms, allow_zero_draft=False:
                         min(mb / ms, mb - mb + 1) if ms else mb - mb + 1),
    "S with the sign flipped": ("residual_mass", lambda p, mb, ms: np.maximum(ms - p * mb, 0).sum()),
}


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_planted_mistakes_fail(monkeypatch, name):
    """Plant a mistake in the oracle: the exact enumeration must reject it."""
    attr, fn = MUTATIONS[name]
    monkeypatch.setattr(tv, attr, fn)
    ok = True
    for shape, V in SHAPES[:3]:
        try:
            ok = ok and _lossless(shape, V, 1)
        except (ZeroDivisionError, InvalidTree, ValueError):
            ok = False
    assert not ok


# ------------------------------------------------------------ P5 ----------

@pytest.mark.parametrize("seed", [5, 6, 7])
def test_chain_expected_length_closed_form(seed):
    """Theorem 2 (Appendix B): on a chain, E[tau] = E_alpha[sum_l p_ini(alpha_l)]
    exactly, and it is at least the E[tau] of token-by-token verification."""
    V = 3
    shape = [-1, 0, 1, 2]
    t = rational_table(V, 3, seed)
    s = rational_table(V, 3, seed + 1000)
    e_tv = 0
    e_closed = 0
    e_token = 0
    for tokens, prob in enumerate_draft_trees(shape, s, V):
        pre = node_prefixes(shape, tokens)
        law = outcome_law(shape, tokens, lambda i: t[pre[i]].copy(),
                          lambda i: s[pre[i]].copy(), V)
        for (a, _), q in law.items():
            e_tv += prob * q * len(pre[a])
        # closed form: p_ini along the chain
        p = F(1)
        tok_acc = F(1)
        for l in range(1, len(shape)):
            x = tokens[l]
            ratio = t[pre[l - 1]][x] / s[pre[l - 1]][x]
            p = min(p * ratio, F(1))
            e_closed += prob * p
            tok_acc = tok_acc * min(ratio, F(1))
            e_token += prob * tok_acc
    assert e_tv == e_closed
    assert e_tv >= e_token


# ------------------------------------------------------------ P6 ----------

@pytest.mark.parametrize("p0", [F(1, 3), F(3, 4)])
@pytest.mark.parametrize("shape,V", SHAPES[:3])
def test_lemma2_subtree_self_similarity(shape, V, p0):
    """Lemma 2 (Appendix A): run on a sub-tree whose root carries rate p0, the
    verifier accepts within the sub-tree with probability p0 and, given that,
    the continuation follows the target model; with probability 1 - p0 the
    sub-tree's root itself is rejected."""
    t = rational_table(V, 3, 11)
    s = rational_table(V, 3, 1011)
    zl, g = z_law(shape, t, s, V, root_rate=p0)
    tl = target_law(t, V, g)
    assert zl.get(None, 0) == 1 - p0
    assert all(zl.get(z, 0) == p0 * q for z, q in tl.items())


# ------------------------------------------------------------ P8 ----------

def test_invariants_along_random_runs():
    """0 <= p <= 1, rates never grow under Eq. (3) (S <= p), the root keeps
    rate 1, and the updated distributions of Eqs. (1)-(2) sum to 1."""
    V = 4
    rng = np.random.default_rng(0)
    shape = [-1, 0, 0, 1, 1, 2, 2]
    t = rational_table(V, 3, 21, zero_prob=0.2)
    s = rational_table(V, 3, 1021, zero_prob=0.2, min_support=2)
    n_checked = 0
    for tokens, _ in enumerate_draft_trees(shape, s, V):
        pre = node_prefixes(shape, tokens)
        st = TraversalState(shape, tokens, lambda i: t[pre[i]].copy(),
                            lambda i: s[pre[i]].copy(), V)
        while True:
            leaf = st.first_leaf()
            assert st.p[0] == 1
            if leaf == 0 or rng.random() < 0.3:
                break
            par = st.parents[leaf]
            before = st.p[par]
            S = tv.residual_mass(before, st.mb[par], st.ms[par])
            assert 0 <= S <= before
            st.reject(leaf)
            assert 0 <= st.p[par] <= before
            if S > 0:
                assert st.mb[par].sum() == 1
            assert st.ms[par].sum() == 1
            assert all(0 <= x <= 1 for x in st.p if x is not None)
            n_checked += 1
    assert n_checked > 50
