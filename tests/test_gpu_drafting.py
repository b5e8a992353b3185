"""GPU parity of drafting the children without replacement (Definition 1,
tv_draft_children) against the oracle (oracle/drafting.py), through the C ABI.

Every child is compared with the oracle's draw given the GPU's tokens for
its earlier siblings: equal wherever u W is at least 1e-5 W from a step of
the oracle's float64 CDF; at a near-tie the GPU's token must be a token of
positive remaining mass whose CDF interval lies within 1e-5 W of u W.  Near
ties are common (a draw landing among the many tail tokens of mass below
1e-5 is one); a token that differs from the oracle's must be within 1e-6 W,
the bound on the kernel's cumulative sums (float32 sums of 256-token tiles,
relative error below 5e-7, accumulated in float64)."""

import numpy as np
import pytest
import torch

from oracle import drafting
from workloads.synth import get_workload, make_inputs, make_inputs_random_shapes

pytestmark = pytest.mark.gpu
TIE = 1e-5
DIFFER = 1e-6


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


def run(tv, parents, drafts, uniforms):
    B, R = parents.shape
    V = drafts.shape[-1]
    v = tv.Verifier(V, R - 1, B, "fp32", path="three")
    toks = v.draft_children(parents.cuda(), drafts.cuda(), uniforms.cuda())
    torch.cuda.synchronize()
    status = v.status()
    v.close()
    return toks.cpu().numpy(), status


def check(parents, drafts, uniforms, got, trees=None):
    """Child-by-child comparison; returns (draws, ties, differing)."""
    par = parents.numpy()
    dr = drafts.numpy()
    un = uniforms.numpy()
    draws = ties = differ = 0
    for b in (range(par.shape[0]) if trees is None else trees):
        assert got[b, 0] == 0
        kids = {}
        for c in range(1, par.shape[1]):
            p = int(par[b, c])
            earlier = kids.setdefault(p, [])
            prev = [int(got[b, j]) for j in earlier]
            earlier.append(c)
            if prev and prev[-1] < 0:
                assert got[b, c] == -1, (b, c)
                continue
            q = dr[b, p].astype(np.float64)
            y, W, margin = drafting.draw_float(q, prev, float(un[b, c]))
            draws += 1
            g = int(got[b, c])
            if y < 0:
                assert g == -1, (b, c, g)
                continue
            if margin >= TIE:
                assert g == y, (b, c, g, y, margin)
                continue
            ties += 1
            if g != y:
                differ += 1
                assert margin < DIFFER, (b, c, g, y, margin)
            qp = q.copy()
            qp[[t for t in prev if t >= 0]] = 0.0
            assert 0 <= g < len(q) and qp[g] > 0, (b, c, g)
            cdf = np.cumsum(qp)
            target = float(un[b, c]) * W
            lo = cdf[g - 1] if g > 0 else 0.0
            assert lo - TIE * W <= target < cdf[g] + TIE * W, (b, c, g, y)
    return draws, ties, differ


def uniforms_for(B, R, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.rand(B, R, generator=g)


@pytest.mark.parametrize("name", ["tiny", "binary4", "eagle_v32k"])
def test_workloads_all_trees(tv, name):
    w = get_workload(name, batch=256 if name == "tiny" else None)
    inp = make_inputs(w, seed=3, device="cpu")
    u = uniforms_for(*inp.parents.shape, seed=4)
    got, status = run(tv, inp.parents, inp.draft_probs, u)
    assert status == 0
    draws, ties, differ = check(inp.parents, inp.draft_probs, u, got)
    print(f"\n{name}: {draws} draws, {ties} within 1e-5 W of a step, {differ} differ")


def test_eagle_v128k_sampled(tv):
    w = get_workload("eagle_v128k")
    inp = make_inputs(w, seed=5, device="cuda")
    B, R = inp.parents.shape
    u = uniforms_for(B, R, seed=6)
    v = tv.Verifier(w.vocab, R - 1, B, "bf16", path="persistent")
    toks = v.draft_children(inp.parents, inp.draft_probs, u.cuda())
    torch.cuda.synchronize()
    assert v.status() == 0
    v.close()
    trees = list(range(0, B, 16))
    sub = inp.draft_probs[trees].cpu()
    draws, _, _ = check(inp.parents[trees].cpu(), sub, u[trees], toks.cpu().numpy()[trees])
    assert draws == len(trees) * (R - 1)


@pytest.mark.parametrize("V", [1001, 4099, 32001])
def test_ragged_vocabularies(tv, V):
    """V not a multiple of 4 (scalar loads) or of the 256-token tile."""
    w = get_workload("binary4", batch=24, vocab=V)
    inp = make_inputs(w, seed=7, device="cpu")
    u = uniforms_for(*inp.parents.shape, seed=8)
    got, status = run(tv, inp.parents, inp.draft_probs, u)
    assert status == 0
    check(inp.parents, inp.draft_probs, u, got)


def test_wide_and_large_trees(tv):
    """1023 draft nodes: a root with 100 children, a node with 200, one with
    300, the rest random; and random-shape trees of the same size."""
    B, V = 6, 8192
    rng = np.random.default_rng(9)
    wide = [-1] + [0] * 100 + [1] * 200 + [2] * 300
    wide += [int(rng.integers(0, len(wide))) for _ in range(1024 - len(wide))]
    parents = torch.tensor(wide, dtype=torch.int32).expand(B, 1024).contiguous()
    g = torch.Generator().manual_seed(9)
    drafts = torch.softmax(3.0 * torch.randn(B, 1024, V, generator=g), dim=-1)
    u = uniforms_for(B, 1024, seed=10)
    got, status = run(tv, parents, drafts, u)
    assert status == 0
    check(parents, drafts, u, got)
    inp = make_inputs_random_shapes(4, 1023, V, seed=9, device="cpu")
    u = uniforms_for(*inp.parents.shape, seed=10)
    got, status = run(tv, inp.parents, inp.draft_probs, u)
    assert status == 0
    check(inp.parents, inp.draft_probs, u, got)


def test_sparse_rows_and_exhausted_support(tv):
    """Rows with few tokens of positive mass: zero-mass tokens are never
    drawn; a node with more children than positive tokens gets -1 for the
    rest and raises TV_STATUS_DRAFT_EXHAUSTED."""
    B, V = 64, 2048
    parents = torch.tensor([-1, 0, 0, 0, 0, 1, 1, 2], dtype=torch.int32).expand(B, 8).contiguous()
    g = torch.Generator().manual_seed(11)
    drafts = torch.rand(B, 8, V, generator=g)
    keep = torch.rand(B, 8, V, generator=g) < 0.002
    drafts = torch.where(keep, drafts, torch.zeros(()))
    drafts[:, :, 1777] += 0.5                       # at least one positive token per row
    drafts = (drafts / drafts.sum(-1, keepdim=True)).contiguous()
    drafts[0, 0] = 0.0
    drafts[0, 0, [5, 900]] = torch.tensor([0.25, 0.75])   # 2 tokens for 4 children
    u = uniforms_for(B, 8, seed=12)
    got, status = run(tv, parents, drafts, u)
    assert status == 128
    check(parents, drafts, u, got)
    assert sorted(got[0, 1:3].tolist()) == [5, 900] and got[0, 3] == -1 and got[0, 4] == -1


def test_edge_uniforms(tv):
    """u = 0 takes the first token of positive mass, u just below 1 the last."""
    B, V = 4, 3000
    parents = torch.tensor([-1, 0, 0], dtype=torch.int32).expand(B, 3).contiguous()
    drafts = torch.zeros(B, 3, V)
    drafts[:, 0, [17, 400, 2999 - 3]] = torch.tensor([0.2, 0.5, 0.3])
    u = torch.tensor([[0.0, 0.0, 0.0], [0.0, 0.99999994, 0.99999994],
                      [0.0, 0.2, 0.2], [0.0, 0.69, 0.1]])
    got, status = run(tv, parents, drafts, u)
    assert status == 0
    assert got[0, 1:].tolist() == [17, 400]
    assert got[1, 1:].tolist() == [2996, 400]
    check(parents, drafts, u, got)


def test_invalid_trees(tv):
    B, V = 3, 512
    parents = torch.tensor([[-1, 0, 0], [0, 0, 0], [-1, 2, 0]], dtype=torch.int32)
    drafts = torch.full((B, 3, V), 1.0 / V)
    u = uniforms_for(B, 3, seed=13)
    got, status = run(tv, parents, drafts, u)
    assert status == 1
    assert got[1].tolist() == [0, -1, -1] and got[2].tolist() == [0, -1, -1]
    check(parents[:1], drafts[:1], u[:1], got[:1])


def test_level_by_level_gives_the_same_tokens(tv):
    """Drafting the first levels of a tree alone gives the tokens a call on
    the whole tree gives them."""
    w = get_workload("eagle_v32k", batch=16)
    inp = make_inputs(w, seed=14, device="cpu")
    u = uniforms_for(*inp.parents.shape, seed=15)
    full, _ = run(tv, inp.parents, inp.draft_probs, u)
    for n_prefix in (5, 17, 41):
        part, status = run(tv, inp.parents[:, :n_prefix].contiguous(),
                           inp.draft_probs[:, :n_prefix].contiguous(),
                           u[:, :n_prefix].contiguous())
        assert status == 0
        assert np.array_equal(part, full[:, :n_prefix])


def test_drafting_then_verification(tv):
    """Tokens from tv_draft_children are valid draft tokens for the
    verification (distinct siblings of positive draft mass), and the
    verification of them matches the oracle."""
    from oracle.verify import verify_batch
    from tests.parity import assert_rate_budget, compare_batch, to_numpy_inputs
    w = get_workload("eagle_v32k", batch=32)
    inp = make_inputs(w, seed=16, device="cuda")
    B, R = inp.parents.shape
    u = uniforms_for(B, R, seed=17).cuda()
    v = tv.Verifier(w.vocab, R - 1, B, "bf16", path="persistent")
    inp.tokens = v.draft_children(inp.parents, inp.draft_probs, u)
    path, tau, bonus, node_p, stats = v.verify(inp.parents, inp.tokens, inp.logits,
                                               inp.draft_probs, inp.temperature, inp.uniforms,
                                               debug=True)
    torch.cuda.synchronize()
    assert v.status() & ~16 == 0
    v.close()
    par, tok, lg, dp, un = to_numpy_inputs(inp)
    _, _, _, det = verify_batch(par, tok, lg, dp, inp.temperature, un, keep_cdf=True)
    summ = compare_batch(det, path.cpu().numpy(), tau.cpu().numpy(), bonus.cpu().numpy(),
                         node_p.cpu().numpy(), stats.cpu().numpy())
    assert not summ["bad"], summ["bad"][:5]
    assert_rate_budget(summ)
