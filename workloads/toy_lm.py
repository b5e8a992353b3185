"""Toy language models and decoding-tree sampling for the distributional tests.

An input generator only: it draws tables of next-token distributions keyed by
prefix and samples (or enumerates) draft trees from them the way Definition 1
(§3.3) describes -- the children of a node drawn from M_s(.|prefix) without
replacement, in child-index order.  It holds none of the verification
arithmetic and is shared by the CPU oracle tests and the GPU tests.
"""

import itertools
from fractions import Fraction

import numpy as np


def prefixes(vocab, max_len):
    for L in range(max_len + 1):
        yield from itertools.product(range(vocab), repeat=L)


def rational_table(vocab, max_len, seed, zero_prob=0.0, max_weight=9, min_support=1):
    """Exact random distributions: for every prefix of length <= max_len a
    vector of Fractions with small integer weights (some possibly zero, at
    least ``min_support`` positive -- a node drafting k children without
    replacement needs a support of at least k tokens)."""
    rng = np.random.default_rng(seed)
    table = {}
    for pre in prefixes(vocab, max_len):
        w = rng.integers(1, max_weight + 1, size=vocab)
        if zero_prob > 0:
            zero = rng.random(vocab) < zero_prob
            keep = rng.permutation(vocab)[:min_support]
            zero[keep] = False
            w = np.where(zero, 0, w)
        tot = int(w.sum())
        table[pre] = np.array([Fraction(int(x), tot) for x in w], dtype=object)
    return table


def float_table(vocab, max_len, seed, concentration=1.0):
    """Float64 Dirichlet distributions for every prefix of length <= max_len."""
    rng = np.random.default_rng(seed)
    return {pre: rng.dirichlet(np.full(vocab, concentration))
            for pre in prefixes(vocab, max_len)}


def node_prefixes(parents, tokens):
    """Prefix (tuple of drafted tokens, root excluded) of every node."""
    out = [()]
    for i in range(1, len(parents)):
        out.append(out[parents[i]] + (int(tokens[i]),))
    return out


def enumerate_draft_trees(parents, ms_table, vocab, with_replacement=False):
    """Every token assignment of a tree shape with its probability under
    Definition 1: children of a node drawn in index order from its draft
    distribution, without replacement (renormalised over the tokens not yet
    drawn among earlier siblings) or, for the negative control, with it."""
    n = len(parents)
    exact = isinstance(ms_table[()][0], Fraction)

    def rec(i, tokens, pres, prob):
        if i == n:
            yield list(tokens), prob
            return
        par = parents[i]
        ms = ms_table[pres[par]]
        used = [tokens[j] for j in range(1, i) if parents[j] == par]
        left = 1
        if not with_replacement:
            left = 1 - sum(ms[t] for t in used)
        for x in range(vocab):
            if ms[x] == 0 or (not with_replacement and x in used):
                continue
            tokens.append(x)
            pres.append(pres[par] + (x,))
            yield from rec(i + 1, tokens, pres, prob * ms[x] / left)
            tokens.pop()
            pres.pop()

    yield from rec(1, [0], [()], Fraction(1) if exact else 1.0)


def sample_draft_trees(parents, ms_table, vocab, count, seed, with_replacement=False):
    """``count`` independent draft trees of one shape, [count, N+1] int32
    (token of the root row is 0 and unused).  Float tables only."""
    rng = np.random.default_rng(seed)
    n = len(parents)
    out = np.zeros((count, n), dtype=np.int32)
    for b in range(count):
        toks = [0]
        pre = [()]
        for i in range(1, n):
            par = parents[i]
            ms = np.asarray(ms_table[pre[par]], dtype=np.float64).copy()
            if not with_replacement:
                for j in range(1, i):
                    if parents[j] == par:
                        ms[toks[j]] = 0.0
            ms /= ms.sum()
            x = int(rng.choice(vocab, p=ms))
            toks.append(x)
            pre.append(pre[par] + (x,))
        out[b] = toks
    return out


def prefix_code(prefix, vocab):
    """Integer code of a prefix: root 0, child code = parent * (V + 1) + x + 1."""
    c = 0
    for x in prefix:
        c = c * (vocab + 1) + x + 1
    return c


def table_array(table, vocab, max_len):
    """Dense [(V+1)^(max_len+1), V] float64 array of a float table, indexed by
    prefix_code (unused codes hold zeros)."""
    out = np.zeros(((vocab + 1) ** (max_len + 1), vocab))
    for pre, row in table.items():
        out[prefix_code(pre, vocab)] = np.asarray(row, dtype=np.float64)
    return out


def sample_trees_batch(parents, ms_array, vocab, count, rng):
    """Vectorised draw of ``count`` draft trees of one shape (Definition 1,
    children without replacement in index order) from a dense table array.
    Returns (tokens [count, N+1] int64, prefix codes [count, N+1] int64)."""
    n = len(parents)
    tokens = np.zeros((count, n), dtype=np.int64)
    codes = np.zeros((count, n), dtype=np.int64)
    rows = np.arange(count)
    for i in range(1, n):
        par = parents[i]
        probs = ms_array[codes[:, par]].copy()
        for j in range(1, i):
            if parents[j] == par:
                probs[rows, tokens[:, j]] = 0.0
        probs /= probs.sum(axis=1, keepdims=True)
        cdf = np.cumsum(probs, axis=1)
        u = rng.random(count)[:, None]
        x = np.minimum((u >= cdf).sum(axis=1), vocab - 1)
        # never land on a zero-probability token through rounding
        bad = probs[rows, x] == 0
        while bad.any():
            x[bad] = np.argmax(probs[bad] > 0, axis=1)
            bad = probs[rows, x] == 0
        tokens[:, i] = x
        codes[:, i] = codes[:, par] * (vocab + 1) + x + 1
    return tokens, codes


def extend_with_target(first_tokens, mb_array, vocab, length, rng):
    """Complete sequences to ``length`` tokens by sampling the target table:
    ``first_tokens`` is a list (per sample) of the tokens already fixed."""
    count = len(first_tokens)
    out = np.full((count, length), -1, dtype=np.int64)
    code = np.zeros(count, dtype=np.int64)
    for b, toks in enumerate(first_tokens):
        for j, x in enumerate(toks[:length]):
            out[b, j] = x
    for j in range(length):
        need = out[:, j] < 0
        if need.any():
            probs = mb_array[code[need]]
            cdf = np.cumsum(probs, axis=1)
            u = rng.random(int(need.sum()))[:, None] * cdf[:, -1:]
            x = np.minimum((u >= cdf).sum(axis=1), vocab - 1)
            out[need, j] = x
        code = code * (vocab + 1) + out[:, j] + 1
    return out
