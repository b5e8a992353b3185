"""GPU parity: the CUDA path against the CPU oracle on the same seeded inputs
and the same pre-drawn uniforms, element by element (see tests/parity.py for
the comparison rule and tolerances).  All calls go through the C ABI."""

import numpy as np
import pytest
import torch

from oracle.verify import verify_batch
from tests.parity import assert_rate_budget, compare_batch, to_numpy_inputs
from workloads.synth import get_workload, make_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


PATHS = ["persistent", "cluster", "three"]


def run_gpu(tv, inp, debug=True, path="auto"):
    B, R = inp.parents.shape
    V = inp.logits.shape[-1]
    dt = "bf16" if inp.logits.dtype == torch.bfloat16 else "fp32"
    v = tv.Verifier(V, R - 1, B, dt, path=path)
    out = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                   inp.uniforms, debug=debug)
    torch.cuda.synchronize()
    status = v.status()
    v.close()
    return [o.cpu().numpy() for o in out], status


# Near-ties are a property of the inputs alone (the oracle's margins), not of
# the GPU: a test tie needs |u - p| < 1e-5 (about 2e-5 of tests); a bonus tie
# needs u W within 1e-5 W of a CDF step, which happens whenever the draw lands
# on one of the many tail tokens of mass below 1e-5 W (observed: 0-10 % of trees
# on these workloads).  The bounds only catch a workload or oracle gone wrong.
MAX_TEST_TIE_FRAC = 0.01
MAX_BONUS_TIE_FRAC = 0.15


def log_summary(meta, path, summ):
    """One JSON line per comparison, appended to $TV_PARITY_LOG when set."""
    import json
    import os
    dest = os.environ.get("TV_PARITY_LOG")
    if not dest:
        return
    rec = {k: summ[k] for k in ("trees", "exact", "ties", "test_ties", "n_rates", "ill",
                                "floor", "max_kappa", "max_p_rel")}
    rec.update(meta=str(meta), path=path, escapes=summ["escapes"])
    with open(dest, "a") as f:
        f.write(json.dumps(rec, default=float) + "\n")


def check(tv, inp, trees=None, path="auto"):
    (gpath, tau, bonus, node_p, stats), status = run_gpu(tv, inp, path=path)
    if trees is None:
        trees = list(range(inp.parents.shape[0]))
    par, tok, lg, dp, un = to_numpy_inputs(inp, trees)
    _, _, _, det = verify_batch(par, tok, lg, dp, inp.temperature, un, keep_cdf=True)
    det = {trees[k]: r for k, r in det.items()}
    summ = compare_batch(det, gpath, tau, bonus, node_p, stats)
    print(f"\n{inp.meta} [{path}]: trees {summ['trees']} exact {summ['exact']} "
          f"ties {summ['ties']} (tests {summ['test_ties']}) rates {summ['n_rates']} "
          f"max p rel err {summ['max_p_rel']:.2e} escapes {len(summ['escapes'])} "
          f"(ill-conditioned {summ['ill']}, max kappa {summ['max_kappa']:.3g}; "
          f"floor {summ['floor']})")
    for e in summ["escapes"]:
        print(f"  escape: tree {e['tree']} node {e['node']} gpu {e['gpu']!r} oracle "
              f"{e['oracle']!r} rel {e['rel']:.2e} kappa {e['kappa']:.3g} S {e['S']!r}")
    log_summary(inp.meta, path, summ)
    assert not summ["bad"], summ["bad"][:5]
    assert_rate_budget(summ)
    assert summ["test_ties"] <= MAX_TEST_TIE_FRAC * summ["trees"] + 1
    assert summ["ties"] - summ["test_ties"] <= MAX_BONUS_TIE_FRAC * summ["trees"] + 2
    return summ, status


@pytest.mark.parametrize("path", PATHS)
def test_tiny_many_seeds(tv, path):
    """The 7-node, V=64, fp32 tree, 512 draws of logits / tree / uniforms."""
    w = get_workload("tiny", batch=512)
    inp = make_inputs(w, seed=0, device="cuda")
    summ, status = check(tv, inp, path=path)
    assert summ["exact"] >= 0.9 * summ["trees"]
    assert status & ~16 == 0


@pytest.mark.parametrize("name", ["chain8", "binary4"])
@pytest.mark.parametrize("sigma", [0.5, 1.0, 2.0])
@pytest.mark.parametrize("path", ["persistent", "cluster"])
def test_chain_and_binary(tv, name, sigma, path):
    w = get_workload(name, sigma=sigma)
    inp = make_inputs(w, seed=1, device="cuda")
    check(tv, inp, path=path)


@pytest.mark.parametrize("path", PATHS)
def test_eagle_v32k_all_trees(tv, path):
    w = get_workload("eagle_v32k")
    inp = make_inputs(w, seed=2, device="cuda")
    check(tv, inp, path=path)


@pytest.mark.parametrize("path", PATHS)
def test_eagle_v128k_sampled(tv, path):
    """Full batch of 128 trees at V=128256 (the benchmark workload); the
    oracle checks a sample of 12 trees."""
    w = get_workload("eagle_v128k")
    inp = make_inputs(w, seed=3, device="cuda")
    trees = list(range(0, 128, 11))
    check(tv, inp, trees=trees, path=path)


@pytest.mark.parametrize("shape", ["4,8,3", "4,4,3", "4,2,2", "8,2,4", "8,1,3", "4,1,2"])
def test_fused_launch_shapes(tv, shape, monkeypatch):
    """Every launch shape of the fused kernel (consumer warps per CTA, CTAs per
    tree, ring stages) gives the oracle's results (V=32000, EAGLE trees)."""
    monkeypatch.setenv("TV_FUSED_PLAN", shape)
    w = get_workload("eagle_v32k", batch=24)
    inp = make_inputs(w, seed=24, device="cuda")
    v = tv.Verifier(w.vocab, w.nodes, 24, "bf16", path="cluster")
    got = v.launch_shape(24, w.nodes)
    v.close()
    ncw, c, st = (int(x) for x in shape.split(","))
    assert got == (1, c, ncw, st)
    check(tv, inp, path="cluster")


@pytest.mark.parametrize("plan", ["4,2,0,0,0", "4,3,0,0,0", "8,2,0,0,0", "4,0,4096,8192,2048"])
def test_persistent_launch_shapes(tv, plan, monkeypatch):
    """Other launch shapes of the persistent kernel (TV_FLOW_PLAN: consumer
    warps, ring stages, pass / normaliser / smallest slice tokens) give the
    oracle's results: three 18 KB stages (three CTAs per SM), eight consumer
    warps, and slices small enough for several per row (V=32000, EAGLE trees)."""
    monkeypatch.setenv("TV_FLOW_PLAN", plan)
    w = get_workload("eagle_v32k", batch=24)
    inp = make_inputs(w, seed=25, device="cuda")
    v = tv.Verifier(w.vocab, w.nodes, 24, "bf16", path="persistent")
    path, _, warps, stages = v.launch_shape(24, w.nodes)
    v.close()
    ncw, st = (int(x) for x in plan.split(",")[:2])
    assert path == 2 and warps == ncw and (st == 0 or stages == st)
    check(tv, inp, path="persistent")


@pytest.mark.parametrize("V,N,want", [(32000, 60, 1), (49152, 127, 1), (32000, 200, 2),
                                       (50000, 60, 2), (128256, 60, 2), (1003, 60, 0)])
def test_auto_path_choice(tv, V, N, want):
    """A handle that picks its path itself: the cluster kernel for short rows
    (V <= 49152, N + 1 <= 128), the persistent kernel otherwise, the
    three-kernel path when V % 8 != 0 (tv_launch_shape's path codes 1, 2, 0)."""
    v = tv.Verifier(V, N, 64, "bf16")
    path, _, _, _ = v.launch_shape(64, N)
    v.close()
    assert path == want


@pytest.mark.parametrize("batch", [1, 8, 40, 400, 1000])
@pytest.mark.parametrize("path", ["persistent", "cluster"])
def test_default_launch_shapes(tv, batch, path):
    """Batch sizes that select different default cluster shapes (clusters of
    8, 8 and 1 CTA, 4 or 8 consumer warps) and, for the persistent kernel,
    fewer and more trees than CTAs."""
    w = get_workload("eagle_v32k", batch=batch)
    inp = make_inputs(w, seed=batch, device="cuda")
    trees = list(range(0, batch, max(1, batch // 40)))
    check(tv, inp, trees=trees, path=path)


def test_eagle_v128k_large_batch_sampled(tv):
    """1024 trees of 128256 tokens: the persistent kernel's largest slices
    (32768 tokens, several per row), sampled trees against the oracle."""
    w = get_workload("eagle_v128k", batch=1024)
    inp = make_inputs(w, seed=9, device="cuda")
    check(tv, inp, trees=list(range(0, 1024, 64)), path="persistent")


@pytest.mark.parametrize("path", PATHS)
def test_margins_reported_by_the_gpu(tv, path):
    """tv_verify_batch_debug's out_margin: the smallest |eta - p| of each
    tree's tests and the bonus draw's distance to the nearer CDF step
    (relative to W), computed on the GPU, against the oracle's float64
    margins within 1e-6 wherever both took the same decisions."""
    w = get_workload("eagle_v32k", batch=64)
    inp = make_inputs(w, seed=41, device="cuda")
    B, R = inp.parents.shape
    v = tv.Verifier(w.vocab, R - 1, B, "bf16", path=path)
    gpath, tau, bonus, node_p, stats, margin = v.verify(
        inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature, inp.uniforms,
        debug=True, margins=True)
    torch.cuda.synchronize()
    v.close()
    tau, bonus, margin = tau.cpu().numpy(), bonus.cpu().numpy(), margin.cpu().numpy()
    stats = stats.cpu().numpy()
    par, tok, lg, dp, un = to_numpy_inputs(inp)
    _, otau, obonus, det = verify_batch(par, tok, lg, dp, inp.temperature, un)
    compared = 0
    for b in range(B):
        r = det[b]
        same_tests = tau[b] == otau[b] and int(stats[b, 0]) == len(r["tests"])
        if same_tests:
            assert abs(float(margin[b, 0]) - r["test_margin"]) <= 1e-6, (b, margin[b], r)
            if bonus[b] == obonus[b]:
                assert abs(float(margin[b, 1]) - r["bonus_margin"]) <= 1e-6, (b, margin[b])
                compared += 1
            else:
                assert margin[b, 1] < 1e-5 and r["bonus_margin"] < 1e-5
        else:
            assert r["test_margin"] < 1e-5 and margin[b, 0] < 1e-5
    assert compared >= B - 4
    near = int(((margin[:, 0] < 1e-5) | (margin[:, 1] < 1e-5)).sum())
    want = sum(1 for b in range(B) if min(det[b]["test_margin"], det[b]["bonus_margin"]) < 1e-5)
    assert abs(near - want) <= 1
    # an invalid tree reports NaN margins
    inp.parents[3, 2] = 5
    v = tv.Verifier(w.vocab, R - 1, B, "bf16", path=path)
    *_, margin2 = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs,
                           inp.temperature, inp.uniforms, debug=True, margins=True)
    torch.cuda.synchronize()
    v.close()
    m2 = margin2.cpu().numpy()
    assert np.isnan(m2[3]).all() and not np.isnan(m2[[0, 1, 2, 4]]).any()


@pytest.mark.parametrize("sigma", [0.5, 2.0])
@pytest.mark.parametrize("batch", [256, 1024])
@pytest.mark.parametrize("name", ["sweep26", "sweep60", "sweep120"])
def test_throughput_sweep_sampled(tv, name, batch, sigma):
    """The V = 151936 throughput sweep (26-, 60- and 120-node trees, 256 and
    1024 trees, draft noise 0.5 and 2) on the default persistent kernel, at
    the batch sizes it is timed at; 12 trees spread over the batch are
    checked against the oracle.  The seed differs per case."""
    w = get_workload(name, batch=batch, sigma=sigma)
    seed = 100 + 10 * ["sweep26", "sweep60", "sweep120"].index(name) + int(sigma) + batch // 256
    inp = make_inputs(w, seed=seed, device="cuda")
    trees = list(range(0, batch, batch // 12))[:12]
    check(tv, inp, trees=trees, path="auto")
    del inp
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["sweep60", "sweep120"])
def test_throughput_sweep_cluster(tv, name):
    """The same sweep trees on the cluster-per-tree path (256 trees, noise 2)."""
    w = get_workload(name, batch=256, sigma=2.0)
    inp = make_inputs(w, seed=77, device="cuda")
    check(tv, inp, trees=list(range(0, 256, 32)), path="cluster")
    del inp
    torch.cuda.empty_cache()


@pytest.mark.parametrize("V", [1000, 1003, 257, 8, 8200, 16392])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("path", ["auto", "cluster"])
def test_ragged_vocab(tv, V, dtype, path):
    """Vocabularies that are not a multiple of the 8-element chunk or of the
    256-element bonus tile exercise the scalar-load path and the tails."""
    from workloads.synth import Workload
    w = Workload("ragged", 48, V, levels=(2, 3, 2), branching=(2, 2, 1),
                 logit_dtype=dtype, sigma=1.0)
    inp = make_inputs(w, seed=V, device="cuda")
    check(tv, inp, path=path)


def test_root_only_trees(tv):
    from workloads.synth import Workload
    w = Workload("root_only", 32, 5000, parents=(-1,), logit_dtype=torch.bfloat16)
    inp = make_inputs(w, seed=5, device="cuda")
    (path, tau, bonus, node_p, stats), status = run_gpu(tv, inp)
    par, tok, lg, dp, un = to_numpy_inputs(inp)
    _, otau, obonus, det = verify_batch(par, tok, lg, dp, inp.temperature, un)
    assert (tau == 0).all()
    near = np.array([det[b]["bonus_margin"] < 1e-5 for b in range(32)])
    assert (bonus[~near] == obonus[~near]).all()


@pytest.mark.parametrize("T", [0.2, 2.0])
def test_temperatures(tv, T):
    from workloads.synth import Workload
    w = Workload("temp", 24, 4096, levels=(3, 6, 6, 4), branching=(3, 2, 1, 1),
                 logit_dtype=torch.bfloat16, temperature=T)
    inp = make_inputs(w, seed=int(T * 10), device="cuda")
    check(tv, inp)


@pytest.mark.parametrize("path", PATHS)
def test_invalid_trees_flagged(tv, path):
    from workloads.synth import Workload
    w = Workload("inv", 6, 512, levels=(2, 2), branching=(2, 1), logit_dtype=torch.float32)
    inp = make_inputs(w, seed=9, device="cuda")
    inp.parents[1, 2] = 3            # parent after child
    inp.tokens[2, 2] = inp.tokens[2, 1]   # duplicate siblings
    inp.tokens[3, 4] = 512           # outside the vocabulary
    inp.parents[4, 0] = 0            # root with a parent
    par = inp.parents[5].tolist()
    inp.draft_probs[5, par[1], inp.tokens[5, 1]] = 0.0   # zero draft probability
    (acc_path, tau, bonus, node_p, stats), status = run_gpu(tv, inp, path=path)
    assert tau[0] >= 0
    assert (tau[1:] == -1).all() and (bonus[1:] == -1).all() and (acc_path[1:] == -1).all()
    assert status & 1 and status & 2 and status & 4 and status & 8
    p2, t2, l2, d2, u2 = to_numpy_inputs(inp)
    _, otau, _, _ = verify_batch(p2, t2, l2, d2, inp.temperature, u2)
    assert (otau[1:] == -1).all()


def test_host_entry_point_matches_device(tv):
    """From host buffers: the same paths and lengths as the device entry point;
    the bonus tokens drawn at accepted leaves in the second phase (a kernel of
    its own) equal the oracle's outside the near-tie band."""
    for name, dt in (("binary4", "fp32"), ("eagle_v32k", "bf16")):
        w = get_workload(name, batch=8)
        inp = make_inputs(w, seed=4, device="cuda")
        (path, tau, bonus, _, stats), _ = run_gpu(tv, inp)
        B, R = inp.parents.shape
        v = tv.Verifier(w.vocab, R - 1, B, dt)
        hp = [inp.parents.cpu(), inp.tokens.cpu(), inp.logits.cpu(), inp.draft_probs.cpu(),
              inp.uniforms.cpu()]
        out = (torch.empty(B, R - 1, dtype=torch.int32), torch.empty(B, dtype=torch.int32),
               torch.empty(B, dtype=torch.int32))
        v.verify_host(hp[0], hp[1], hp[2], hp[3], inp.temperature, hp[4], out)
        v.close()
        assert (out[0].numpy() == path).all() and (out[1].numpy() == tau).all()
        par, tok, lg, dp, un = to_numpy_inputs(inp)
        _, _, obonus, det = verify_batch(par, tok, lg, dp, inp.temperature, un)
        for b in range(B):
            if det[b]["bonus_margin"] >= 1e-5 and det[b]["test_margin"] >= 1e-5:
                assert int(out[2][b]) == int(obonus[b]), (name, b)
        assert stats[:, 3].sum() > 0   # some trees ended at an accepted leaf


@pytest.mark.parametrize("shapes", ["same", "random"])
def test_host_entry_point_copies_only_needed_draft_rows(tv, shapes):
    """The host entry point copies the logit and draft rows of nodes with
    children, then the logit rows of the accepted leaves only (2-D copies when
    all trees share a shape, per tree otherwise).  Two calls
    on one handle with different inputs: stale staging from the first would
    change the second's results if a needed row were missed."""
    from workloads.synth import make_inputs_random_shapes
    if shapes == "same":
        mk = lambda seed: make_inputs(get_workload("eagle_v32k", batch=24), seed=seed,
                                      device="cuda")
    else:
        mk = lambda seed: make_inputs_random_shapes(24, 60, 32000, seed=seed, device="cuda")
    first, second = mk(51), mk(52)
    B, R = second.parents.shape
    v = tv.Verifier(32000, R - 1, B, "bf16")
    out = (torch.empty(B, R - 1, dtype=torch.int32), torch.empty(B, dtype=torch.int32),
           torch.empty(B, dtype=torch.int32))
    for inp in (first, second):
        hp = [x.cpu() for x in (inp.parents, inp.tokens, inp.logits, inp.draft_probs,
                                inp.uniforms)]
        v.verify_host(hp[0], hp[1], hp[2], hp[3], inp.temperature, hp[4], out)
    h2d, d2h = v.last_host_copy_bytes()
    want = v.verify(second.parents, second.tokens, second.logits, second.draft_probs,
                    second.temperature, second.uniforms, debug=True)
    torch.cuda.synchronize()
    assert v.status() & ~16 == 0
    v.close()
    for a, b in zip(out[:2], want[:2]):
        assert torch.equal(a, b.cpu())
    # bonus tokens: the draws at accepted leaves come from the second phase's
    # own kernel, equal to the device path's away from a CDF step
    leaf = want[4][:, 3].cpu().numpy() > 0
    same = out[2].numpy() == want[2].cpu().numpy()
    assert same[~leaf].all() and same[leaf].mean() > 0.8
    par = second.parents.cpu().numpy()
    internal = sum(len({int(p) for p in par[b, 1:]}) for b in range(B))
    n_leaf = int(leaf.sum())
    V = 32000
    assert h2d == (2 * B * R * 4 + B * (R + 1) * 4 + internal * V * (2 + 4) + n_leaf * V * 2 +
                   n_leaf * 8)
    assert d2h == B * (R - 1) * 4 + 2 * B * 4 + (B * 4 if n_leaf else 0)


def test_host_argument_errors(tv):
    w = get_workload("tiny", batch=2)
    inp = make_inputs(w, seed=0, device="cuda")
    v = tv.Verifier(64, 7, 2, "fp32")
    with pytest.raises(tv.LibraryError) as e:
        v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, 0.0, inp.uniforms)
    assert e.value.code == -2
    with pytest.raises(tv.LibraryError) as e:
        v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, float("nan"),
                 inp.uniforms)
    assert e.value.code == -2
    v.close()
    small = tv.Verifier(64, 3, 2, "fp32")
    rc = small.lib.tv_verify_batch(small.handle, 2, 7, None, None, None, None, 1.0, None,
                                   None, None, None, None)
    assert rc == -4
    rc = small.lib.tv_verify_batch(small.handle, 1, 3, None, None, None, None, 1.0, None,
                                   None, None, None, None)
    assert rc == -1
    rc = small.lib.tv_verify_batch(small.handle, 0, 3, None, None, None, None, 1.0, None,
                                   None, None, None, None)
    assert rc == 0
    small.close()
