"""Host logic of bench.py: the algorithmic byte count and the guard that keeps
a stale ncu traffic figure out of the roofline."""

import os
import shutil

import pytest
import torch

import bench


def test_algorithmic_bytes_counts_rows_passes_and_bonus():
    V, lb = 1000, 2
    # columns: tests, passes, distinct rows passed, bonus from a leaf, rows normalised
    stats = torch.tensor([[3, 2, 1, 0, 4],    # residual bonus
                          [1, 0, 0, 1, 2],    # leaf bonus
                          [0, 0, 0, 0, 0]],   # invalid tree
                         dtype=torch.int32)
    tau = torch.tensor([1, 2, -1], dtype=torch.int32)
    # trees with 5, 3 and 3 internal rows (rows 0..4 / 0..2 have children)
    parents = torch.tensor([[-1, 0, 1, 2, 3, 4, 0],
                            [-1, 0, 1, 2, 0, 0, 0],
                            [-1, 0, 1, 2, 0, 0, 0]], dtype=torch.int32)
    ab = bench.algorithmic_bytes(stats, tau, parents, V, lb)
    # unique: normalised target rows, draft rows of nodes with passes, leaf row
    assert ab["unique"] == (4 + 2) * V * lb + 1 * V * 4 + 1 * V * lb
    # eager count A: every internal row, R draft rows, the leaf row
    assert ab["s8d"] == (5 + 3) * V * lb + 1 * V * 4 + 1 * V * lb
    # re-read inclusive: each pass streams both rows again, bonus one row
    passes = 2 * V * (lb + 4)
    bonus = V * (lb + 4) + V * lb
    assert ab["reread"] == (4 + 2) * V * lb + passes + bonus
    assert ab["normaliser"] == (4 + 2) * V * lb
    assert ab["R_per_tree"] == 0.5 and ab["passes_per_tree"] == 1.0
    assert ab["internal_rows_per_tree"] == 4.0


def _copy_tree(tmp_path):
    root = tmp_path / "repo"
    shutil.copytree(os.path.join(bench.ROOT, "paper_2505_12398_gb300", "csrc"),
                    root / "paper_2505_12398_gb300" / "csrc")
    shutil.copytree(os.path.join(bench.ROOT, "profiles"), root / "profiles")
    return root


def test_kernel_traffic_follows_the_source_hash(tmp_path, monkeypatch):
    """A profile's DRAM figure is used only while the kernel sources hash to
    the value recorded with it."""
    root = _copy_tree(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(root))
    prof = root / "profiles" / "launches_testload_B7_persistent.md"
    prof.write_text("# test\n\n    kernel-sources-sha256: "
                    + bench.kernel_sources_sha256() + "\n    dram-bytes-per-launch: 12345\n")
    assert bench.kernel_traffic("testload", 7) == 12345
    assert bench.kernel_traffic("testload", 8) is None   # no profile of that batch
    src = root / "paper_2505_12398_gb300" / "csrc" / "tv_flow.cu"
    src.write_text(src.read_text() + "\n// changed\n")
    assert bench.kernel_traffic("testload", 7) is None


def test_lmhead_oracle_leg_matches_the_oracle_on_the_generated_logits(tmp_path):
    """The CPU leg of the LM-head pipeline (oracle logits from the dumped
    bf16 operands, then Algorithm 3) reaches the tau the oracle gives on the
    generator's own logits (exact operands here, so both hold the same
    logits)."""
    import numpy as np
    from oracle.verify import verify_tree
    from workloads.synth import get_workload, make_lmhead_inputs
    w = get_workload("binary4", batch=3, vocab=1024, logit_dtype=torch.bfloat16)
    lin = make_lmhead_inputs(w, hidden=64, seed=4)
    # operands k/16 and a bias column of integers: every product is exact
    g = torch.Generator().manual_seed(9)
    lin.hidden.copy_((torch.randint(-8, 9, lin.hidden.shape, generator=g) / 16.0).to(torch.bfloat16))
    lin.weight.copy_((torch.randint(-8, 9, lin.weight.shape, generator=g) / 16.0).to(torch.bfloat16))
    inp = lin.inputs
    B, R = inp.parents.shape
    inp.logits.copy_((lin.hidden.float() @ lin.weight.float().T).view(B, R, -1).to(torch.bfloat16))
    d = bench.dump_lmhead_sample(lin, range(B), str(tmp_path))
    with bench._oracle_pool(2) as pool:
        _, n, taus = bench.time_lmhead_oracle(d, B, inp.temperature, pool)
    assert n == B
    for b in range(B):
        r = verify_tree(inp.parents[b].numpy(), inp.tokens[b].numpy(),
                        inp.logits[b].float().numpy().astype(np.float64),
                        inp.draft_probs[b].numpy(), inp.temperature, inp.uniforms[b].numpy())
        assert taus[b] == r["tau"]


def test_full_pipeline_oracle_leg_drafts_first(tmp_path):
    """With drafting uniforms in the sample, the CPU leg drafts each tree with
    the drafting oracle before verifying it."""
    import numpy as np
    from oracle.drafting import sample_tree
    from oracle.verify import verify_tree
    from workloads.synth import get_workload, make_lmhead_inputs
    w = get_workload("binary4", batch=3, vocab=512, logit_dtype=torch.bfloat16)
    lin = make_lmhead_inputs(w, hidden=64, seed=5)
    g = torch.Generator().manual_seed(10)
    lin.hidden.copy_((torch.randint(-8, 9, lin.hidden.shape, generator=g) / 16.0).to(torch.bfloat16))
    lin.weight.copy_((torch.randint(-8, 9, lin.weight.shape, generator=g) / 16.0).to(torch.bfloat16))
    inp = lin.inputs
    B, R = inp.parents.shape
    inp.logits.copy_((lin.hidden.float() @ lin.weight.float().T).view(B, R, -1).to(torch.bfloat16))
    u_draft = torch.rand(B, R, generator=g)
    d = bench.dump_lmhead_sample(lin, range(B), str(tmp_path), u_draft)
    with bench._oracle_pool(2) as pool:
        _, n, taus = bench.time_lmhead_oracle(d, B, inp.temperature, pool)
    for b in range(B):
        drafts = inp.draft_probs[b].numpy()
        toks = sample_tree(inp.parents[b].numpy(), drafts, u_draft[b].tolist())
        r = verify_tree(inp.parents[b].numpy(), np.asarray(toks),
                        inp.logits[b].float().numpy().astype(np.float64), drafts,
                        inp.temperature, inp.uniforms[b].numpy())
        assert taus[b] == r["tau"]
