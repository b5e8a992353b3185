"""Pins of the drafting oracle (oracle/drafting.py, Definition 1: children
drawn without replacement in child order) against the independent statement
of Definition 1's law in workloads/toy_lm.py, numpy's searchsorted, and
invariants."""

from fractions import Fraction

import numpy as np
import pytest
from scipy import stats

from oracle import drafting
from workloads.toy_lm import enumerate_draft_trees

Q4 = [Fraction(3, 10), Fraction(0), Fraction(1, 2), Fraction(1, 5)]      # a zero-mass token
Q5 = [Fraction(1, 7), Fraction(2, 7), Fraction(1, 14), Fraction(5, 14), Fraction(1, 7)]


def conditional_law(q, k):
    """P(token of child j | tokens of children 0..j-1) from Definition 1's
    enumerated law of ordered k-tuples (a depth-1 tree with k children)."""
    parents = [-1] + [0] * k
    law = {tuple(t[1:]): p for t, p in enumerate_draft_trees(parents, {(): q}, len(q))}
    marg = {}
    for tup, p in law.items():
        for j in range(k + 1):
            marg[tup[:j]] = marg.get(tup[:j], Fraction(0)) + p
    return lambda prefix, t: marg.get(prefix + (t,), Fraction(0)) / marg[prefix]


def intervals(cond, prefix, V):
    """[lo, hi) of u giving each token after ``prefix``, from the law."""
    out, lo = {}, Fraction(0)
    for t in range(V):
        p = cond(prefix, t)
        if p > 0:
            out[t] = (lo, lo + p)
            lo += p
    assert lo == 1
    return out


def probe_all(q, k, sampler):
    """For every prefix the law allows and every next token of positive
    probability: the sampler returns that token at the lower end of its
    u-interval and just below the upper end, and the previous token just
    below the lower end."""
    V = len(q)
    cond = conditional_law(q, k)

    def rec(prefix, us):
        if len(prefix) == k:
            return
        iv = intervals(cond, prefix, V)
        toks = sorted(iv)
        for n, t in enumerate(toks):
            lo, hi = iv[t]
            eps = Fraction(1, 10 ** 12)
            assert sampler(q, len(prefix) + 1, us + [lo])[-1] == t
            assert sampler(q, len(prefix) + 1, us + [hi - eps])[-1] == t
            if n > 0:
                assert sampler(q, len(prefix) + 1, us + [lo - eps])[-1] == toks[n - 1]
            rec(prefix + (t,), us + [(lo + hi) / 2])

    rec((), [])


@pytest.mark.parametrize("q,k", [(Q4, 1), (Q4, 2), (Q4, 3), (Q5, 3), (Q5, 5)])
def test_partition_of_u_is_definition_1_law_exactly(q, k):
    """Exact: the oracle's map u -> token splits [0, 1) into intervals of
    exactly Definition 1's conditional probabilities, in token order, at
    every draw -- so its law of ordered k-tuples is Definition 1's."""
    probe_all(q, k, drafting.sample_children)


def test_planted_mistakes_fail_the_partition_pin(monkeypatch):
    """Negative controls, planted in the oracle: siblings drawn with
    replacement, or the remaining mass not renormalised."""
    orig = drafting.draw_without_replacement
    monkeypatch.setattr(drafting, "draw_without_replacement",
                        lambda q, removed, u: orig(q, [], u))
    with pytest.raises(AssertionError):
        probe_all(Q5, 3, drafting.sample_children)
    monkeypatch.setattr(drafting, "draw_without_replacement", orig)

    def unnormalised(q, removed, u):
        t, W = orig(q, removed, u)
        # compares u (not u * W) with the cumulative sums of the remaining mass
        cdf = Fraction(0)
        for y in range(len(q)):
            cdf += Fraction(0) if y in removed else q[y]
            if u < cdf:
                return y, W
        return -1, W
    monkeypatch.setattr(drafting, "draw_without_replacement", unnormalised)
    with pytest.raises(AssertionError):
        probe_all(Q5, 3, drafting.sample_children)


def test_single_draw_is_searchsorted():
    """k = 1 is plain inverse-CDF sampling: numpy's searchsorted on the
    cumulative sums (side='right': the smallest y with u W < CDF(y))."""
    rng = np.random.default_rng(0)
    for _ in range(200):
        V = int(rng.integers(2, 300))
        q = rng.dirichlet(np.full(V, 0.3)).astype(np.float32).astype(np.float64)
        q[rng.random(V) < 0.2] = 0.0
        if q.sum() == 0:
            continue
        for u in rng.random(5):
            want = int(np.searchsorted(np.cumsum(q), u * q.sum(), side="right"))
            want = min(want, int(np.flatnonzero(q)[-1]))
            assert drafting.sample_children(list(q), 1, [float(u)]) == [want]


def test_ordered_tuples_chi_square():
    """Monte Carlo on float64: the frequencies of ordered 3-tuples from V = 6
    follow Definition 1's enumerated law."""
    rng = np.random.default_rng(1)
    qf = rng.dirichlet(np.ones(6))
    q = [Fraction(x).limit_denominator(10 ** 9) for x in qf]
    s = sum(q)
    q = [x / s for x in q]
    law = {tuple(t[1:]): p for t, p in enumerate_draft_trees([-1, 0, 0, 0], {(): q}, 6)}
    keys = sorted(law)
    n = 30000
    counts = dict.fromkeys(keys, 0)
    qfl = [float(x) for x in q]
    for u in rng.random((n, 3)):
        counts[tuple(drafting.sample_children(qfl, 3, list(u)))] += 1
    obs = np.array([counts[k] for k in keys])
    exp = np.array([float(law[k]) * n for k in keys])
    assert stats.chisquare(obs, exp).pvalue > 1e-3


def test_tree_samples_each_parent_separately():
    """Siblings are drawn from their own parent's row with only their own
    earlier siblings removed: sample_tree equals sample_children per parent;
    siblings are distinct and of positive mass."""
    rng = np.random.default_rng(2)
    parents = [-1, 0, 0, 0, 1, 1, 2, 4, 4, 4]
    V = 12
    for _ in range(50):
        drafts = rng.dirichlet(np.full(V, 0.5), size=len(parents))
        drafts[rng.random(drafts.shape) < 0.3] = 0.0
        drafts[:, 0] += 1e-3                         # keep mass in every row
        u = list(rng.random(len(parents)))
        toks = drafting.sample_tree(parents, drafts, u)
        for p in set(parents[1:]):
            kids = [c for c in range(1, len(parents)) if parents[c] == p]
            want = drafting.sample_children(list(drafts[p]), len(kids), [u[c] for c in kids])
            assert [toks[c] for c in kids] == want
            got = [toks[c] for c in kids if toks[c] >= 0]
            assert len(set(got)) == len(got)
            assert all(drafts[p][t] > 0 for t in got)


def test_more_children_than_support():
    q = [0.0, 0.5, 0.0, 0.5]
    assert drafting.sample_children(q, 4, [0.1, 0.9, 0.5, 0.5]) == [1, 3, -1, -1]
    assert drafting.sample_tree([-1, 0, 0, 0], [q, q, q, q], [0, 0.7, 0.2, 0.3]) == [0, 3, 1, -1]


def test_margin_and_invalid_trees():
    q = [0.25, 0.25, 0.5]
    assert drafting.draw_float(q, [], 0.3)[::2] == (1, pytest.approx(0.05))
    assert drafting.draw_float(q, [1], 0.5)[::2] == (2, pytest.approx(1 / 6))
    for bad in ([0, 0, 0], [-1, 1, 0], [-1, 0, 3]):
        assert drafting.sample_tree(bad, [q] * 3, [0.0, 0.5, 0.5]) == [0, -1, -1]


def test_float_path_matches_exact_path():
    """The float64 draw (numpy cumulative sums) agrees with the exact
    Fraction draw on dyadic rows, where float64 sums are exact."""
    rng = np.random.default_rng(3)
    for _ in range(300):
        V = int(rng.integers(2, 40))
        w = rng.integers(0, 9, V)
        if w.sum() == 0:
            continue
        qf = [Fraction(int(x), 64) for x in w]
        removed = [int(x) for x in rng.choice(V, int(rng.integers(0, V)), replace=False)]
        u = Fraction(int(rng.integers(0, 2 ** 20)), 2 ** 20)
        assert drafting.draw_float([float(x) for x in qf], removed, float(u))[0] == \
            drafting.draw_without_replacement(qf, removed, u)[0]
