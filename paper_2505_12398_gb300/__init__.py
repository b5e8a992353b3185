"""Batched Traversal Verification on GB300 (arXiv 2505.12398).

Thin Python binding of the C ABI in ``include/tv.h``: argument marshalling
only.  Every step of the verification runs in the CUDA kernels of
``libtv.so`` (built in-tree by ``paper_2505_12398_gb300.build``); there is no
CPU path, and using the binding without the compiled library raises.

    v = Verifier(vocab=32000, max_nodes=60, max_batch=64, logit_dtype="bf16")
    path, tau, bonus = v.verify(parents, tokens, logits, draft_probs, 1.0, uniforms)
"""

from ._binding import (PATH_FLAGS, TV_BF16, TV_FP32, TV_STATUS, LibraryError, Verifier,
                       library, library_path, status_names)

__all__ = ["Verifier", "library", "library_path", "LibraryError", "PATH_FLAGS", "TV_BF16",
           "TV_FP32", "TV_STATUS", "status_names"]
