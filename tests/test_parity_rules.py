"""The comparison rules of tests/parity.py, checked on the CPU: GPU-shaped
outputs are built from the oracle's own results on a small batch, then
perturbed on purpose, and each rule must accept or reject exactly what it
states (rates within 1e-5 relative; escapes only within the float32
cancellation bound or the absolute floor, and only in a budgeted number of
trees; bit-exact paths, tau and bonus away from near-ties; invalid and pruned
nodes marked as the library marks them)."""

import copy

import numpy as np
import pytest

from oracle.verify import verify_batch
from tests.parity import (K_EPS, P_ATOL, P_EQ0, P_RTOL, assert_rate_budget, compare_batch,
                          escape_budget, to_numpy_inputs)
from workloads.synth import get_workload, make_inputs


@pytest.fixture(scope="module")
def oracle_batch():
    w = get_workload("tiny", batch=64)
    inp = make_inputs(w, seed=11, device="cpu")
    par, tok, lg, dp, un = to_numpy_inputs(inp)
    _, _, _, det = verify_batch(par, tok, lg, dp, inp.temperature, un, keep_cdf=True)
    return det, par.shape


def gpu_like(det, shape):
    """The arrays tv_verify_batch_debug would return if it matched the oracle
    to float32 rounding."""
    B, R = shape
    g_path = np.full((B, R - 1), -1, dtype=np.int32)
    g_tau = np.full(B, -1, dtype=np.int32)
    g_bonus = np.full(B, -1, dtype=np.int32)
    g_p = np.full((B, R), np.nan, dtype=np.float32)
    g_stats = np.zeros((B, 7), dtype=np.int32)
    for b, r in det.items():
        if "invalid" in r:
            continue
        g_tau[b] = r["tau"]
        g_path[b, :r["tau"]] = r["path"]
        g_bonus[b] = r["bonus"]
        for node, _, p in r["tests"]:
            g_p[b, node] = np.float32(p)
        for c in r["pruned"]:
            g_p[b, c] = 0.0
        g_stats[b, :4] = [sum(1 for _, _, p in r["tests"] if p >= P_EQ0), r["n_passes"],
                          len(r["rejected_at"]), int(r["leaf_row_read"])]
    return g_path, g_tau, g_bonus, g_p, g_stats


def untied(det):
    """Trees without a near-tie, with at least one tested rate above the
    absolute floor (the rates the relative rule governs)."""
    out = []
    for b, r in det.items():
        if "invalid" in r or r["bonus_margin"] < 1e-5:
            continue
        tests = [(k, t) for k, t in enumerate(r["tests"]) if abs(t[1] - t[2]) >= 1e-5]
        if len(tests) == len(r["tests"]) and any(t[2] > 1e-3 for _, t in tests):
            out.append(b)
    return out


def first_big_test(r):
    return next(k for k, (_, _, p) in enumerate(r["tests"]) if p > 1e-3)


def test_the_oracle_against_itself_is_exact(oracle_batch):
    det, shape = oracle_batch
    summ = compare_batch(det, *gpu_like(det, shape))
    assert not summ["bad"]
    assert summ["escapes"] == []
    assert summ["max_p_rel"] < 1e-7            # float32 storage of the rates only
    assert summ["exact"] == summ["trees"] - summ["ties"]
    assert_rate_budget(summ)


def test_rates_within_the_bar_pass_and_beyond_it_fail_unless_explained(oracle_batch):
    det, shape = oracle_batch
    b = untied(det)[0]
    k = first_big_test(det[b])
    node, _, p = det[b]["tests"][k]
    g = gpu_like(det, shape)
    # 0.5e-5 relative: inside the bar
    g[3][b, node] = p * (1 + 0.5 * P_RTOL)
    summ = compare_batch(det, *g)
    assert not summ["bad"] and summ["escapes"] == []
    # 3e-5 relative with kappa 1: outside every bound -> a failure
    d1 = copy.deepcopy(det)
    d1[b]["kappa_at_test"] = [1.0] * len(d1[b]["tests"])
    g[3][b, node] = p * (1 + 3 * P_RTOL)
    summ = compare_batch(d1, *g)
    assert summ["bad"] and summ["bad"][0][0] == b
    # the same error with kappa 100: within K_EPS * kappa -> an escape, listed
    d2 = copy.deepcopy(det)
    d2[b]["kappa_at_test"] = [100.0] * len(d2[b]["tests"])
    assert 3 * P_RTOL <= K_EPS * 100.0
    summ = compare_batch(d2, *g)
    assert not summ["bad"]
    assert [(e["tree"], e["node"]) for e in summ["escapes"]] == [(b, node)]
    assert summ["ill"] == 1 and summ["max_p_rel"] > 2 * P_RTOL   # the true maximum
    assert_rate_budget(summ)


def test_a_small_rate_escapes_only_through_the_absolute_floor(oracle_batch):
    det, shape = oracle_batch
    b = untied(det)[0]
    k = first_big_test(det[b])
    node, u, _ = det[b]["tests"][k]
    d = copy.deepcopy(det)
    d[b]["kappa_at_test"] = [1.0] * len(d[b]["tests"])
    tiny = 1e-9 if u > 1e-3 else 0.5
    d[b]["tests"][k] = (node, u, tiny)
    g = gpu_like(d, shape)
    g[3][b, node] = tiny * 1.001                  # 1e-3 relative, 1e-12 absolute
    summ = compare_batch(d, *g)
    assert not summ["bad"] and summ["floor"] == 1
    g[3][b, node] = tiny + 2 * P_ATOL             # past the floor too
    summ = compare_batch(d, *g)
    assert summ["bad"]


def test_escape_budget_counts_trees_against_compared_rates(oracle_batch):
    det, shape = oracle_batch
    trees = untied(det)
    assert len(trees) >= 4
    d = copy.deepcopy(det)
    g = gpu_like(d, shape)
    for b in trees:
        d[b]["kappa_at_test"] = [100.0] * len(d[b]["tests"])
    summ0 = compare_batch(d, *g)
    allowed = escape_budget(summ0["n_rates"])
    assert allowed == 2 + summ0["n_rates"] // 50
    for n_esc in (allowed, allowed + 1):
        if n_esc > len(trees):
            continue
        gg = [x.copy() for x in g]
        for b in trees[:n_esc]:
            node, _, p = d[b]["tests"][first_big_test(d[b])]
            gg[3][b, node] = p * (1 + 3 * P_RTOL)
        summ = compare_batch(d, *gg)
        assert not summ["bad"]
        if n_esc <= allowed:
            assert_rate_budget(summ)
        else:
            with pytest.raises(AssertionError):
                assert_rate_budget(summ)


def test_paths_tau_and_bonus_are_bit_exact_away_from_ties(oracle_batch):
    det, shape = oracle_batch
    b = untied(det)[0]
    for field, bad_value in (("tau", None), ("bonus", None)):
        g = gpu_like(det, shape)
        if field == "tau":
            g[1][b] = det[b]["tau"] + 1
        else:
            g[2][b] = det[b]["bonus"] + 1
        summ = compare_batch(det, *g)
        assert [x[0] for x in summ["bad"]] == [b], field
    g = gpu_like(det, shape)
    if det[b]["tau"] > 0:
        g[0][b, 0] = g[0][b, 0] + 1
        assert compare_batch(det, *g)["bad"]


def test_a_near_tie_is_counted_and_not_compared_past(oracle_batch):
    det, shape = oracle_batch
    b = untied(det)[0]
    d = copy.deepcopy(det)
    node, u, p = d[b]["tests"][0]
    d[b]["tests"][0] = (node, p + 0.5e-5, p)     # |u - p| below the tie margin
    g = gpu_like(d, shape)
    g[1][b] = d[b]["tau"] + 1                     # the GPU went the other way at the tie
    g[2][b] = d[b]["bonus"] + 1
    summ = compare_batch(d, *g)
    assert not summ["bad"]
    assert summ["test_ties"] >= 1


def test_invalid_and_pruned_nodes_are_marked_like_the_library(oracle_batch):
    det, shape = oracle_batch
    d = copy.deepcopy(det)
    b = untied(det)[0]
    d[b] = {"invalid": "planted"}
    g = gpu_like(d, shape)
    assert not compare_batch(d, *g)["bad"]        # tau, bonus, path all -1
    g[1][b] = 0
    assert compare_batch(d, *g)["bad"]
    pr = [b2 for b2, r in det.items() if "invalid" not in r and r["pruned"]
          and not any(abs(t[1] - t[2]) < 1e-5 for t in r["tests"])]
    if pr:
        b2 = pr[0]
        g = gpu_like(det, shape)
        g[3][b2, det[b2]["pruned"][0]] = 0.25     # a removed node reported with a rate
        assert compare_batch(det, *g)["bad"]
