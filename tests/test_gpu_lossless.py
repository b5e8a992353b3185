"""Losslessness of the CUDA path (Theorem 1 via Lemma 1), by Monte Carlo.

A prefix-keyed toy language model drives 10^6 draft trees per case through
the kernels; each output (X^tau, Y) is extended to gamma_max tokens with the
target model and the empirical law of Z^{gamma_max} is compared with
prod_j M_b(z_j | z_<j) by a chi-square test.  A negative control (the same
trees verified with a wrong target, so the output law is not M_b) must fail.
"""

import itertools

import numpy as np
import pytest
import scipy.stats
import torch

from workloads.toy_lm import (extend_with_target, float_table, sample_trees_batch,
                              table_array)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


def z_counts(tv, shape, V, count, seed, wrong_target=False, method="traversal", path="auto"):
    rng = np.random.default_rng(seed)
    L = 4
    tb = float_table(V, L, seed, concentration=0.8)
    ts = float_table(V, L, seed + 1, concentration=0.8)
    mb = table_array(tb, V, L)
    ms = table_array(ts, V, L)
    tokens, codes = sample_trees_batch(shape, ms, V, count, rng)
    n = len(shape)
    depth = [0] * n
    for i in range(1, n):
        depth[i] = depth[shape[i]] + 1
    g = max(depth)
    mb_used = mb
    if wrong_target:
        mb_used = mb.copy()
        mb_used[0] = np.roll(mb_used[0], 1)   # the root's target is not the model's
    with np.errstate(divide="ignore"):
        logits = np.log(mb_used[codes]).astype(np.float32)
    drafts = ms[codes].astype(np.float32)
    dev = torch.device("cuda")
    par = torch.tensor(shape, dtype=torch.int32).expand(count, n).contiguous().to(dev)
    tok = torch.from_numpy(tokens.astype(np.int32)).to(dev)
    lg = torch.from_numpy(logits).to(dev)
    dp = torch.from_numpy(drafts).to(dev)
    un = torch.rand(count, n + 1, generator=torch.Generator(device=dev).manual_seed(seed),
                    device=dev)
    v = tv.Verifier(V, n - 1, count, "fp32", method=method, path=path)
    path, tau, bonus = v.verify(par, tok, lg, dp, 1.0, un)
    torch.cuda.synchronize()
    status = v.status()
    v.close()
    assert status & ~16 == 0
    path = path.cpu().numpy()
    tau = tau.cpu().numpy()
    bonus = bonus.cpu().numpy()
    assert (tau >= 0).all()
    first = []
    for b in range(count):
        toks = [int(tokens[b, j]) for j in path[b, :tau[b]]]
        if tau[b] < g:
            toks.append(int(bonus[b]))
        first.append(toks)
    z = extend_with_target(first, mb, V, g, rng)
    cells = list(itertools.product(range(V), repeat=g))
    idx = np.zeros(count, dtype=np.int64)
    for j in range(g):
        idx = idx * V + z[:, j]
    obs = np.bincount(idx, minlength=V ** g).astype(np.float64)
    exp = np.array([np.prod([tb[c[:j]][c[j]] for j in range(g)]) for c in cells])
    return obs, exp


def chi2_p(obs, exp):
    n = obs.sum()
    keep = exp * n >= 5
    o = np.append(obs[keep], obs[~keep].sum())
    e = np.append(exp[keep], exp[~keep].sum()) * n
    if e[-1] == 0:
        o, e = o[:-1], e[:-1]
    return scipy.stats.chisquare(o, e).pvalue


@pytest.mark.parametrize("shape,V,path", [([-1, 0, 0, 1, 1, 2, 2], 4, "auto"),
                                          ([-1, 0, 0, 0, 1, 1, 2, 4], 3, "auto"),
                                          ([-1, 0, 1, 2], 8, "persistent"),
                                          ([-1, 0, 0, 1, 1, 2, 2], 8, "cluster")])
def test_kernel_output_law_is_target(tv, shape, V, path):
    """V = 3 and 4 take the three-kernel path (V % 8 != 0); V = 8 runs the
    persistent kernel and the cluster kernel."""
    obs, exp = z_counts(tv, shape, V, 1_000_000, seed=V * 17 + len(shape), path=path)
    assert chi2_p(obs, exp) > 1e-3


def test_negative_control_detects_wrong_law(tv):
    obs, exp = z_counts(tv, [-1, 0, 0, 1, 1, 2, 2], 4, 1_000_000, seed=5, wrong_target=True)
    assert chi2_p(obs, exp) < 1e-6


@pytest.mark.parametrize("shape", [[-1, 0, 0, 1, 1, 2, 2], [-1, 0, 1, 2]])
def test_token_level_output_law_is_target(tv, shape):
    """The token-level verifier (TV_FLAG_TOKEN_LEVEL) is lossless too."""
    obs, exp = z_counts(tv, shape, 8, 1_000_000, seed=101 + len(shape), method="token")
    assert chi2_p(obs, exp) > 1e-3
