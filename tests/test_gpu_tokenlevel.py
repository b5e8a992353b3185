"""GPU parity of the token-level verifier (TV_FLAG_TOKEN_LEVEL): the CUDA path
against the oracle's top-down verifier on the same seeded inputs and uniforms,
with the comparison rule of tests/parity.py.  All calls go through the C ABI."""

import pytest
import torch

from oracle.tokenlevel import verify_batch_token_level
from tests.parity import TIE, assert_rate_budget, compare_batch, to_numpy_inputs
from workloads.synth import get_workload, make_inputs

pytestmark = pytest.mark.gpu

PATHS = ["persistent", "cluster"]


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


def summ_tie(r):
    """A near-tie lets the two sides walk different paths past it."""
    return any(abs(u - p) < TIE for _, u, p in r["tests"])


def check(tv, inp, path, trees=None, max_tie_frac=0.25):
    B, R = inp.parents.shape
    V = inp.logits.shape[-1]
    dt = "bf16" if inp.logits.dtype == torch.bfloat16 else "fp32"
    v = tv.Verifier(V, R - 1, B, dt, path=path, method="token")
    out = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                   inp.uniforms, debug=True)
    torch.cuda.synchronize()
    status = v.status()
    v.close()
    g_path, g_tau, g_bonus, g_p, g_stats = [o.cpu().numpy() for o in out]
    if trees is None:
        trees = list(range(B))
    par, tok, lg, dp, un = to_numpy_inputs(inp, trees)
    _, _, _, det = verify_batch_token_level(par, tok, lg, dp, inp.temperature, un,
                                            keep_cdf=True)
    det = {trees[k]: r for k, r in det.items()}
    summ = compare_batch(det, g_path, g_tau, g_bonus, g_p, g_stats)
    print(f"\n{inp.meta} token-level {path}: trees {summ['trees']} exact {summ['exact']} "
          f"ties {summ['ties']} max p rel err {summ['max_p_rel']:.2e} "
          f"ill-conditioned {summ['ill']}")
    assert not summ["bad"], summ["bad"][:5]
    assert_rate_budget(summ)
    assert summ["ties"] <= max_tie_frac * summ["trees"] + 1
    # rows normalised: exactly the internal nodes the walk entered (the root
    # and every accepted internal node); an accepted leaf's row is only
    # read by the bonus draw
    for b, r in det.items():
        if "invalid" not in r and not summ_tie(r):
            internal = set(r["internal"])
            want = sum(1 for i in r["rows_read"] if i in internal)
            assert int(g_stats[b][4]) == want, (b, int(g_stats[b][4]), want)
    return summ, status


@pytest.mark.parametrize("path", PATHS)
def test_tiny_many_seeds(tv, path):
    w = get_workload("tiny", batch=512)
    inp = make_inputs(w, seed=10, device="cuda")
    summ, status = check(tv, inp, path)
    assert summ["exact"] >= 0.9 * summ["trees"]
    assert status & ~16 == 0


@pytest.mark.parametrize("name", ["chain8", "binary4"])
@pytest.mark.parametrize("sigma", [0.5, 2.0])
def test_chain_and_binary(tv, name, sigma):
    w = get_workload(name, sigma=sigma)
    inp = make_inputs(w, seed=11, device="cuda")
    check(tv, inp, "persistent")


@pytest.mark.parametrize("path", PATHS)
def test_eagle_v32k_all_trees(tv, path):
    w = get_workload("eagle_v32k")
    inp = make_inputs(w, seed=12, device="cuda")
    check(tv, inp, path)


def test_eagle_v128k_sampled(tv):
    w = get_workload("eagle_v128k")
    inp = make_inputs(w, seed=13, device="cuda")
    check(tv, inp, "persistent", trees=list(range(0, 128, 11)))


@pytest.mark.parametrize("batch", [1, 1000])
def test_fewer_and_more_trees_than_ctas(tv, batch):
    w = get_workload("eagle_v32k", batch=batch)
    inp = make_inputs(w, seed=14 + batch, device="cuda")
    check(tv, inp, "persistent", trees=list(range(0, batch, max(1, batch // 40))))


def test_token_level_needs_a_single_kernel_path(tv):
    with pytest.raises(tv.LibraryError):
        tv.Verifier(32000, 8, 4, "bf16", path="three", method="token")
    with pytest.raises(tv.LibraryError):
        tv.Verifier(1003, 8, 4, "fp32", method="token")     # V % 8 != 0


def test_same_inputs_traversal_accepts_at_least_as_much_on_average(tv):
    """Not a per-tree property (the two methods spend the uniforms on
    different nodes), but Traversal Verification's mean accepted length on a
    batch of EAGLE trees is not below the token-level verifier's."""
    w = get_workload("eagle_v32k", batch=2048)
    inp = make_inputs(w, seed=15, device="cuda")
    taus = {}
    for method in ("traversal", "token"):
        v = tv.Verifier(w.vocab, w.nodes, 2048, "bf16", method=method)
        _, tau, _ = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs,
                             inp.temperature, inp.uniforms)
        taus[method] = tau.float().mean().item()
        v.close()
    print(f"\nmean tau: traversal {taus['traversal']:.3f} token-level {taus['token']:.3f}")
    assert taus["traversal"] >= taus["token"] - 0.1
