"""CUDA graphs: drafting, the LM head and verification captured into one graph
and replayed on new inputs written into the same buffers give what the
same calls give eagerly; the persistent kernel is never captured."""

import pytest
import torch

from workloads.synth import get_workload, make_lmhead_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


def test_draft_lmhead_verify_graph_replays(tv):
    w = get_workload("eagle_v32k", batch=16)
    lin = make_lmhead_inputs(w, hidden=256, seed=21, device="cuda")
    inp = lin.inputs
    B, R = inp.parents.shape
    N, V, T = R - 1, w.vocab, inp.temperature
    g = torch.Generator(device="cuda").manual_seed(22)
    u_draft = torch.rand(B, R, generator=g, device="cuda")
    vg = tv.Verifier(V, N, B, "bf16")                         # picks its path itself
    ve = tv.Verifier(V, N, B, "bf16", path="cluster")        # eager reference, same kernel
    tok = torch.empty(B, R, dtype=torch.int32, device="cuda")
    logits = torch.empty(B, R, V, dtype=torch.bfloat16, device="cuda")
    stats = torch.empty(B * R, 2, dtype=torch.float32, device="cuda")
    outs = [torch.empty(B, N, dtype=torch.int32, device="cuda"),
            torch.empty(B, dtype=torch.int32, device="cuda"),
            torch.empty(B, dtype=torch.int32, device="cuda")]

    def pipeline(v):
        v.draft_children(inp.parents, inp.draft_probs, u_draft, out=tok)
        v.lm_head(lin.hidden, lin.weight, T, out=(logits.view(B * R, V), stats))
        v.verify(inp.parents, tok, logits, inp.draft_probs, T, inp.uniforms, out=outs)

    pipeline(vg)                      # first calls outside the capture
    pipeline(ve)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        pipeline(vg)
    for round_ in range(3):
        if round_:
            # new inputs in the captured buffers
            u_draft.copy_(torch.rand(B, R, generator=g, device="cuda"))
            inp.uniforms.copy_(torch.rand(B, R + 1, generator=g, device="cuda"))
            lin.hidden.copy_((torch.randn(B * R, 256, generator=g, device="cuda")).to(torch.bfloat16))
        graph.replay()
        torch.cuda.synchronize()
        got = [t.clone() for t in (tok, logits, stats, *outs)]
        pipeline(ve)
        torch.cuda.synchronize()
        want = [t.clone() for t in (tok, logits, stats, *outs)]
        for a, b in zip(got, want):
            assert torch.equal(a, b)
    assert vg.status() & ~16 == 0 and ve.status() & ~16 == 0
    vg.close()
    ve.close()


def test_persistent_handle_refuses_capture(tv):
    w = get_workload("binary4", batch=4, vocab=1024, logit_dtype=torch.bfloat16)
    from workloads.synth import make_inputs
    inp = make_inputs(w, seed=23, device="cuda")
    B, R = inp.parents.shape
    v = tv.Verifier(1024, R - 1, B, "bf16", path="persistent")
    v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, 1.0, inp.uniforms)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        with pytest.raises(tv.LibraryError):
            v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, 1.0, inp.uniforms)
    v.close()
