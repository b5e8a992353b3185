"""Property-based pins of the oracles (hypothesis): losslessness of Traversal
Verification and of the token-level verifier in exact arithmetic on random
tree shapes, Definition 1's law for the drafting oracle on random rows, and
the bf16 rounding of the LM-head oracle."""

from fractions import Fraction

import numpy as np
import pytest

hyp = pytest.importorskip("hypothesis")
st = pytest.importorskip("hypothesis.strategies")
from hypothesis import given, settings  # noqa: E402

from oracle import drafting, lmhead  # noqa: E402
from oracle.exact import target_law, z_law  # noqa: E402
from tests.test_oracle_drafting import probe_all  # noqa: E402
from workloads.toy_lm import rational_table  # noqa: E402


@st.composite
def trees(draw, max_nodes=6):
    n = draw(st.integers(1, max_nodes))
    parents = [-1]
    for i in range(1, n + 1):
        parents.append(draw(st.integers(0, i - 1)))
    return parents


def depth(parents):
    d = [0] * len(parents)
    for i in range(1, len(parents)):
        d[i] = d[parents[i]] + 1
    return max(d)


@settings(max_examples=60, deadline=None)
@given(trees(), st.integers(2, 3), st.integers(0, 10 ** 6), st.sampled_from([0.0, 0.3]))
def test_lossless_on_random_shapes(parents, V, seed, zero_prob):
    """Theorem 1 exactly: for any tree shape, the law of Z^{gamma_max}
    (every draft tree, every accept / reject branch, rational arithmetic)
    is the target model's law."""
    branching = max(parents[1:].count(i) for i in range(len(parents)))
    if branching > V:
        return                                  # more siblings than tokens: no valid tree
    L = depth(parents)                          # rows for every prefix up to the leaves
    t = rational_table(V, L, seed, zero_prob=zero_prob)
    s = rational_table(V, L, seed + 1, zero_prob=zero_prob, min_support=branching)
    zl, g = z_law(parents, t, s, V)
    tl = target_law(t, V, g)
    assert set(zl) <= set(tl)
    assert all(zl.get(z, 0) == q for z, q in tl.items())


@settings(max_examples=40, deadline=None)
@given(trees(), st.integers(2, 3), st.integers(0, 10 ** 6))
def test_token_level_lossless_on_random_shapes(parents, V, seed):
    """The token-level verifier (the comparator) is lossless too, on any
    shape."""
    from oracle import tokenlevel
    branching = max(parents[1:].count(i) for i in range(len(parents)))
    if branching > V:
        return
    L = depth(parents)
    t = rational_table(V, L, seed)
    s = rational_table(V, L, seed + 1, min_support=branching)
    zl, g = z_law(parents, t, s, V, outcome=tokenlevel.outcome_law)
    tl = target_law(t, V, g)
    assert set(zl) <= set(tl)
    assert all(zl.get(z, 0) == q for z, q in tl.items())


@settings(max_examples=40, deadline=None)
@given(st.lists(st.integers(0, 6), min_size=2, max_size=6), st.integers(1, 4))
def test_drafting_partition_on_random_rows(weights, k):
    """The drafting oracle's u-intervals are Definition 1's conditional
    probabilities at every draw, on random rows (zeros allowed)."""
    positive = sum(1 for w in weights if w > 0)
    if positive == 0:
        return
    k = min(k, positive)
    total = sum(weights)
    q = [Fraction(w, total) for w in weights]
    probe_all(q, k, drafting.sample_children)


@settings(max_examples=60, deadline=None)
@given(st.lists(st.integers(0, 9), min_size=2, max_size=8), st.integers(1, 5),
       st.lists(st.floats(0.0, 0.999999), min_size=5, max_size=5))
def test_drafting_prefix_and_support(weights, k, us):
    """Tokens are distinct and of positive mass, and drafting k children
    gives the first k - 1 of them when drafting k - 1 (siblings are drawn in
    order, each from what its earlier siblings left)."""
    if sum(weights) == 0:
        return
    q = [w / sum(weights) for w in weights]
    toks = drafting.sample_children(q, k, us)
    got = [t for t in toks if t >= 0]
    assert len(set(got)) == len(got) and all(q[t] > 0 for t in got)
    assert toks[:k - 1] == drafting.sample_children(q, k - 1, us)
    assert (len(got) == min(k, sum(1 for w in weights if w > 0)))


@settings(max_examples=200, deadline=None)
@given(st.floats(-1e30, 1e30, allow_nan=False, allow_infinity=False))
def test_bf16_rounding_properties(x):
    """Idempotent, within half a bf16 step of the value, and exactly a value
    with 8 significant bits."""
    r = float(lmhead.to_bf16(x))
    assert float(lmhead.to_bf16(r)) == r
    if x != 0.0:
        e = np.frexp(x)[1]
        assert abs(r - x) <= np.ldexp(1.0, e - 9)
        m, er = np.frexp(r)
        assert m * 256.0 == np.rint(m * 256.0)


@settings(max_examples=50, deadline=None)
@given(st.lists(st.floats(-50, 50, allow_nan=False), min_size=2, max_size=40))
def test_bf16_rounding_is_monotone(xs):
    xs = np.sort(np.asarray(xs, dtype=np.float64))
    r = lmhead.to_bf16(xs)
    assert np.all(np.diff(r) >= 0)
