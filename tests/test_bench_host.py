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
    rows, other = bench.algorithmic_bytes(stats, tau, V, lb)
    assert rows == (4 + 2) * V * lb
    passes = 2 * V * (lb + 4)
    bonus = V * (lb + 4) + V * lb
    assert other == passes + bonus


def _copy_tree(tmp_path):
    root = tmp_path / "repo"
    shutil.copytree(os.path.join(bench.ROOT, "paper_2505_12398_gb300", "csrc"),
                    root / "paper_2505_12398_gb300" / "csrc")
    shutil.copytree(os.path.join(bench.ROOT, "profiles"), root / "profiles")
    return root


def test_kernel_traffic_follows_the_source_hash(tmp_path, monkeypatch):
    prof = os.path.join(bench.ROOT, "profiles", "launches_eagle_v128k_B128_persistent.md")
    if not os.path.exists(prof):
        pytest.skip("no committed launch profile")
    root = _copy_tree(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(root))
    got = bench.kernel_traffic("eagle_v128k", 128)
    if got is None:
        pytest.skip("the committed profile predates the current kernel sources")
    assert got > 0
    assert bench.kernel_traffic("eagle_v128k", 64) is None   # no profile of that batch
    src = root / "paper_2505_12398_gb300" / "csrc" / "tv_flow.cu"
    src.write_text(src.read_text() + "\n// changed\n")
    assert bench.kernel_traffic("eagle_v128k", 128) is None
