"""Failure detection on the GPU without a fault: the persistent kernel's
bounded waits run out when a job is never published (tv_debug_withhold_job),
the call ends through the kernel's abort path with TV_STATUS_TIMEOUT, and the
handle keeps working."""

import time

import pytest
import torch

from workloads.synth import get_workload, make_inputs

pytestmark = pytest.mark.gpu

TIMEOUT = 32


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


def _call(v, inp):
    out = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                   inp.uniforms)
    torch.cuda.synchronize()
    return [o.clone() for o in out]


def test_withheld_job_times_out_and_the_handle_recovers(tv):
    w = get_workload("eagle_v32k", batch=8)
    inp = make_inputs(w, seed=77, device="cuda")
    v = tv.Verifier(w.vocab, w.nodes, 8, "bf16", path="persistent")
    ref = _call(v, inp)
    assert v.status() & ~16 == 0
    assert (ref[1] >= 0).all()

    v.withhold_job(3)
    t0 = time.perf_counter()
    out = _call(v, inp)
    elapsed = time.perf_counter() - t0
    status = v.status()
    assert status & TIMEOUT
    assert elapsed < 30.0                       # the idle limit is 2 s
    assert out[1][3].item() == -1 and out[2][3].item() == -1
    assert (out[0][3] == -1).all()
    for b in range(8):                          # trees done before the abort are right
        if out[1][b].item() >= 0:
            assert out[1][b].item() == ref[1][b].item()
            assert out[2][b].item() == ref[2][b].item()
            assert torch.equal(out[0][b], ref[0][b])

    again = _call(v, inp)                       # the next call is unaffected
    assert v.status() & ~16 == 0
    for a, r in zip(again, ref):
        assert torch.equal(a, r)
    v.close()


def test_withhold_rejects_a_tree_outside_the_batch(tv):
    v = tv.Verifier(32000, 8, 4, "bf16", path="persistent")
    with pytest.raises(tv.LibraryError):
        v.withhold_job(4)
    with pytest.raises(tv.LibraryError):
        v.withhold_job(-1)
    v.close()
