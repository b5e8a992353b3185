"""GPU parity of the LM head fused with the row normalisers (tv_lm_head,
tcgen05 tensor cores) and of verification with given normalisers
(tv_verify_batch_stats), against the oracle.  All calls go through the C ABI."""

import numpy as np
import pytest
import torch

from oracle import lmhead
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


def _run(tv, H, W, T):
    M, K = H.shape
    V = W.shape[0]
    v = tv.Verifier(V, 7, (M + 7) // 8, "bf16", path="persistent")
    lg, st = v.lm_head(H.cuda(), W.cuda(), T)
    torch.cuda.synchronize()
    assert v.status() == 0
    v.close()
    return lg.float().cpu().numpy().astype(np.float64), st.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("M,K,V", [(128, 64, 256), (300, 256, 1000), (700, 4096, 32000)])
def test_exact_operands(tv, M, K, V):
    """Operands k/16 with |k| <= 8: every product and partial sum is exact in
    fp32, so the stored logits must equal the oracle's bf16 rounding bit for
    bit, and the normalisers must agree on every row."""
    g = torch.Generator().manual_seed(M * 7 + K)
    H = (torch.randint(-8, 9, (M, K), generator=g).float() / 16).to(torch.bfloat16)
    W = (torch.randint(-8, 9, (V, K), generator=g).float() / 16).to(torch.bfloat16)
    T = 0.8
    got, st = _run(tv, H, W, T)
    ref = lmhead.to_bf16(lmhead.logits(H.float().numpy(), W.float().numpy()))
    assert np.array_equal(got, ref)
    m, s = lmhead.row_stats(ref, T)
    assert np.array_equal(st[:, 0], m)
    assert np.max(np.abs(st[:, 1] - s) / s) < 1e-5


@pytest.mark.parametrize("M,K,V", [(300, 256, 1000), (256, 4096, 8192)])
def test_random_operands(tv, M, K, V):
    """Random operands: an entry may round the other way only where the fp32
    accumulation error bound K 2^-24 sum_k |h_k w_k| reaches a bf16 rounding
    boundary; rows without such an entry have the oracle's normaliser."""
    g = torch.Generator().manual_seed(M + K + V)
    H = (torch.randn(M, K, generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(V, K, generator=g) * 0.5).to(torch.bfloat16)
    T = 1.0
    got, st = _run(tv, H, W, T)
    h, w = H.float().numpy(), W.float().numpy()
    exact = lmhead.logits(h, w)
    ref = lmhead.to_bf16(exact)
    mag = lmhead.logits(np.abs(h), np.abs(w))
    bound = 2 * K * 2.0 ** -24 * mag + 2.0 ** -23 * np.abs(exact)
    unsure = lmhead.bf16_boundary_distance(exact) < bound
    differ = got != ref
    assert not (differ & ~unsure).any()
    assert differ.mean() < 0.01
    # the worst-case bound above covers every entry once K is large; a tighter
    # one still far above fp32 accumulation error (about 2^-24 per add of a
    # partial sum) but far below what a dropped or repeated K block or a wrong
    # column would cause: |stored - exact| <= half a bf16 step + 2^-16 sum|hw|
    half = np.ldexp(1.0, np.frexp(got)[1] - 9)
    tight = half + 2.0 ** -16 * mag
    assert np.all(np.abs(got - exact) <= tight)
    rows = ~differ.any(axis=1)
    if rows.any():
        m, s = lmhead.row_stats(ref[rows], T)
        assert np.array_equal(st[rows, 0], m)
        assert np.max(np.abs(st[rows, 1] - s) / s) < 1e-5


def test_lm_head_argument_errors(tv):
    v = tv.Verifier(1000, 7, 8, "bf16", path="persistent")
    H = torch.zeros(16, 100, dtype=torch.bfloat16, device="cuda")     # K % 64 != 0
    W = torch.zeros(1000, 100, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(tv.LibraryError):
        v.lm_head(H, W, 1.0)
    v.close()


@pytest.mark.parametrize("name", ["eagle_v32k", "binary4"])
def test_verification_with_given_normalisers(tv, name):
    """Row normalisers given by the caller (here computed in float64 from the
    stored logits): the persistent kernel reads no row for a normaliser and
    matches the oracle."""
    w = get_workload(name)
    inp = make_inputs(w, seed=41, device="cuda")
    B, R = inp.parents.shape
    V = inp.logits.shape[-1]
    lf = inp.logits.double()
    m = lf.max(dim=-1).values
    s = torch.exp2((lf - m[..., None]) * (lmhead.LOG2E / inp.temperature)).sum(dim=-1)
    row_stats = torch.stack([m, s], dim=-1).float().contiguous()
    dt = "bf16" if inp.logits.dtype == torch.bfloat16 else "fp32"
    v = tv.Verifier(V, R - 1, B, dt, path="persistent")
    path, tau, bonus, node_p, stats = v.verify_stats(
        inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature, inp.uniforms,
        row_stats, debug=True)
    torch.cuda.synchronize()
    assert v.status() & ~16 == 0
    v.close()
    assert (stats[:, 4] == 0).all()                 # no row streamed for a normaliser
    par, tok, lg, dp, un = to_numpy_inputs(inp)
    _, _, _, det = verify_batch(par, tok, lg, dp, inp.temperature, un, keep_cdf=True)
    summ = compare_batch(det, path.cpu().numpy(), tau.cpu().numpy(), bonus.cpu().numpy(),
                         node_p.cpu().numpy(), stats.cpu().numpy())
    assert not summ["bad"], summ["bad"][:5]
    assert_rate_budget(summ)
    assert summ["ties"] <= 0.25 * summ["trees"] + 1


def test_lm_head_then_verification(tv):
    """The fused pipeline: logits and normalisers from tv_lm_head, then
    verification with them, against the oracle run on the oracle's own
    logits (exact operands, so both sides hold the same logits)."""
    B, N, V, K = 16, 30, 8192, 256
    R = N + 1
    g = torch.Generator().manual_seed(5)
    H = (torch.randint(-8, 9, (B * R, K), generator=g).float() / 16).to(torch.bfloat16)
    Wt = (torch.randint(-8, 9, (V, K), generator=g).float() / 16).to(torch.bfloat16)
    ref = lmhead.to_bf16(lmhead.logits(H.float().numpy(), Wt.float().numpy()))
    T = 1.0
    w = get_workload("binary4", batch=B, vocab=V)
    base = make_inputs(w, seed=6, device="cpu")    # tree shape, uniforms
    logits_ref = torch.from_numpy(ref).float().reshape(B, R, V)
    drafts = torch.softmax((logits_ref + torch.randn(B, R, V, generator=g)) / T, dim=-1)
    # children drawn from the new draft rows without replacement (Gumbel top-k)
    tokens = torch.zeros(B, R, dtype=torch.int64)
    parents = base.parents[0].tolist()
    for i in range(R):
        kids = [c for c in range(1, R) if parents[c] == i]
        if kids:
            keys = torch.log(drafts[:, i]) - torch.log(-torch.log(
                torch.rand(B, V, generator=g).clamp(min=1e-12)))
            tokens[:, kids] = torch.topk(keys, len(kids), dim=-1).indices
    v = tv.Verifier(V, N, B, "bf16", path="persistent")
    lg, st = v.lm_head(H.cuda(), Wt.cuda(), T)
    path, tau, bonus, node_p, stats = v.verify_stats(
        base.parents.cuda(), tokens.int().cuda(), lg.view(B, R, V), drafts.cuda(), T,
        base.uniforms.cuda(), st, debug=True)
    torch.cuda.synchronize()
    assert v.status() & ~16 == 0
    v.close()
    assert np.array_equal(lg.float().cpu().numpy(), ref)
    _, _, _, det = verify_batch(base.parents.numpy(), tokens.numpy(), logits_ref.numpy(),
                                drafts.numpy(), T, base.uniforms.numpy(), keep_cdf=True)
    summ = compare_batch(det, path.cpu().numpy(), tau.cpu().numpy(), bonus.cpu().numpy(),
                         node_p.cpu().numpy(), stats.cpu().numpy())
    assert not summ["bad"], summ["bad"][:5]
    assert_rate_budget(summ)


def test_token_level_with_given_normalisers(tv):
    """The token-level verifier on the given-normaliser kernel matches its
    oracle."""
    from oracle.tokenlevel import verify_batch_token_level
    w = get_workload("eagle_v32k", batch=32)
    inp = make_inputs(w, seed=42, device="cuda")
    B, R = inp.parents.shape
    lf = inp.logits.double()
    m = lf.max(dim=-1).values
    s = torch.exp2((lf - m[..., None]) * (lmhead.LOG2E / inp.temperature)).sum(dim=-1)
    row_stats = torch.stack([m, s], dim=-1).float().contiguous()
    del lf
    v = tv.Verifier(w.vocab, R - 1, B, "bf16", path="persistent", method="token")
    path, tau, bonus, node_p, stats = v.verify_stats(
        inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature, inp.uniforms,
        row_stats, debug=True)
    torch.cuda.synchronize()
    assert v.status() & ~16 == 0
    v.close()
    assert (stats[:, 4] == 0).all()
    par, tok, lg, dp, un = to_numpy_inputs(inp)
    _, _, _, det = verify_batch_token_level(par, tok, lg, dp, inp.temperature, un, keep_cdf=True)
    summ = compare_batch(det, path.cpu().numpy(), tau.cpu().numpy(), bonus.cpu().numpy(),
                         node_p.cpu().numpy(), stats.cpu().numpy())
    assert not summ["bad"], summ["bad"][:5]
    assert_rate_budget(summ)


def test_new_entry_points_argument_errors(tv):
    """Host-side checks of tv_draft_children and tv_verify_batch_stats."""
    import ctypes
    v = tv.Verifier(1000, 7, 4, "bf16", path="three")
    lib, h = v.lib, v.handle
    par = torch.zeros(4, 8, dtype=torch.int32, device="cuda")
    dr = torch.zeros(4, 8, 1000, dtype=torch.float32, device="cuda")
    u = torch.zeros(4, 8, dtype=torch.float32, device="cuda")
    out = torch.zeros(4, 8, dtype=torch.int32, device="cuda")
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    assert lib.tv_draft_children(h, 5, 7, P(par), P(dr), P(u), P(out), None) == \
        -4  # TV_ERR_CAPACITY
    assert lib.tv_draft_children(h, 4, 8, P(par), P(dr), P(u), P(out), None) == \
        -4  # TV_ERR_CAPACITY
    assert lib.tv_draft_children(h, 4, 7, None, P(dr), P(u), P(out), None) == \
        -1  # TV_ERR_INVALID_ARG
    assert lib.tv_draft_children(h, 0, 7, None, None, None, None, None) == 0
    # given normalisers need the persistent kernel
    lg = torch.zeros(4, 8, 1000, dtype=torch.bfloat16, device="cuda")
    st = torch.ones(32, 2, dtype=torch.float32, device="cuda")
    with pytest.raises(tv.LibraryError):
        v.verify_stats(par, out, lg, dr, 1.0, torch.zeros(4, 9, device="cuda"), st)
    v.close()


def test_bench_size_sampled_rows(tv):
    """The bench's launch: 7808 x 4096 x 128256, 61 row tiles walked in two
    groups (32 and a tail of 29).  Exact operands, so sampled rows from both
    groups and the edges of row tiles must equal the oracle bit for bit over
    every column, with their normalisers."""
    M, K, V, B, N = 7808, 4096, 128256, 128, 60
    g = torch.Generator(device="cuda").manual_seed(61)
    H = (torch.randint(-8, 9, (M, K), generator=g, device="cuda") / 16.0).to(torch.bfloat16)
    W = (torch.randint(-8, 9, (V, K), generator=g, device="cuda") / 16.0).to(torch.bfloat16)
    v = tv.Verifier(V, N, B, "bf16", path="persistent")
    lg, st = v.lm_head(H, W, 0.7)
    torch.cuda.synchronize()
    assert v.status() == 0
    v.close()
    rows = [0, 1, 127, 128, 2047, 4095, 4096, 4097, 6000, 7679, 7680, 7807]
    h = H[rows].float().cpu().numpy()
    got = lg[rows].float().cpu().numpy().astype(np.float64)
    st = st[rows].cpu().numpy().astype(np.float64)
    ref = np.empty((len(rows), V))
    Wc = W.float().cpu().numpy()
    for v0 in range(0, V, 16384):
        ref[:, v0:v0 + 16384] = lmhead.logits(h, Wc[v0:v0 + 16384])
    ref = lmhead.to_bf16(ref)
    assert np.array_equal(got, ref)
    m, s = lmhead.row_stats(ref, 0.7)
    assert np.array_equal(st[:, 0], m)
    assert np.max(np.abs(st[:, 1] - s) / s) < 1e-5
