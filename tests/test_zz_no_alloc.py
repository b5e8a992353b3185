"""tv_verify_batch_noalloc: verification without device allocation.

Some callers cannot allocate device memory (a serving process whose pool
reserved the device up front and forbids new allocations, an embedding whose
allocator owns the whole device).  This entry point keeps its
scratch in a fixed static device array instead of a handle's workspace.  Its
results must equal those of the handle-based three-kernel path (the same
kernels run on the same inputs), call after call: the shared array keeps the
previous call's contents and every call must clear what it needs.

Kept in a file of its own, collected last.
"""

import ctypes

import pytest
import torch

from workloads.synth import Workload, get_workload, make_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


def _p(t):
    return ctypes.c_void_p(t.data_ptr())


def noalloc(tv, inp, dtype_code, stream=None):
    B, R = inp.parents.shape
    V = inp.logits.shape[-1]
    out = (torch.full((B, R - 1), -7, dtype=torch.int32, device="cuda"),
           torch.full((B,), -7, dtype=torch.int32, device="cuda"),
           torch.full((B,), -7, dtype=torch.int32, device="cuda"))
    s = stream or torch.cuda.current_stream()
    rc = tv.library().tv_verify_batch_noalloc(
        torch.cuda.current_device(), B, R - 1, V, dtype_code, _p(inp.parents), _p(inp.tokens),
        _p(inp.logits), _p(inp.draft_probs), float(inp.temperature), _p(inp.uniforms),
        _p(out[0]), _p(out[1]), _p(out[2]), ctypes.c_void_p(s.cuda_stream))
    assert rc == 0, tv.library().tv_strerror(rc)
    torch.cuda.synchronize()
    return [o.cpu() for o in out]


def reference(tv, inp, dtype):
    B, R = inp.parents.shape
    v = tv.Verifier(inp.logits.shape[-1], R - 1, B, dtype, path="three")
    out = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                   inp.uniforms)
    torch.cuda.synchronize()
    v.close()
    return [o.cpu() for o in out]


def test_noalloc_matches_handle_path_twice(tv):
    """Two calls in a row (different batches, the second smaller) give exactly
    the handle path's paths, lengths and bonus tokens."""
    first = make_inputs(get_workload("eagle_v32k", batch=48), seed=11, device="cuda")
    second = make_inputs(get_workload("binary4", batch=16), seed=12, device="cuda")
    for inp, code, dt in ((first, tv.TV_BF16, "bf16"), (second, tv.TV_FP32, "fp32"),
                          (first, tv.TV_BF16, "bf16")):
        got = noalloc(tv, inp, code)
        want = reference(tv, inp, dt)
        for g, w in zip(got, want):
            assert torch.equal(g, w)
        assert (got[1] >= 0).all()


def test_noalloc_rejects_oversized_batches(tv):
    """More than 65536 rows do not fit the static scratch: a clear error, no launch."""
    lib = tv.library()
    z = ctypes.c_void_p(0)
    rc = lib.tv_verify_batch_noalloc(0, 1100, 60, 32000, tv.TV_BF16, z, z, z, z, 1.0, z, z, z,
                                     z, z)
    assert rc == -4   # TV_ERR_CAPACITY
    rc = lib.tv_verify_batch_noalloc(0, 4, 7, 64, tv.TV_FP32, z, z, z, z, 0.0, z, z, z, z, z)
    assert rc == -2   # TV_ERR_TEMPERATURE


def test_noalloc_invalid_tree_then_valid(tv):
    """An invalid tree marks only its own outputs; the next call starts clean."""
    w = Workload("inv", 6, 512, levels=(2, 2), branching=(2, 1), logit_dtype=torch.float32)
    inp = make_inputs(w, seed=9, device="cuda")
    inp.parents[2, 2] = 3
    got = noalloc(tv, inp, tv.TV_FP32)
    assert got[1][2] == -1 and (got[1][[0, 1, 3, 4, 5]] >= 0).all()
    inp.parents[2, 2] = 0
    got = noalloc(tv, inp, tv.TV_FP32)
    want = reference(tv, inp, "fp32")
    for g, wv in zip(got, want):
        assert torch.equal(g, wv)
