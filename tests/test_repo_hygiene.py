"""Repository rules that a change could silently break: profile summaries are
short text that gives the commands behind their numbers, no committed file is
named for a round, and nothing committed depends on the ignored working
folder or names the batched copy calls this library never uses."""

import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def committed_files():
    try:
        out = subprocess.run(["git", "ls-files"], cwd=ROOT, capture_output=True, text=True,
                             check=True).stdout
    except (OSError, subprocess.CalledProcessError):
        pytest.skip("not a git checkout")
    return [f for f in out.splitlines() if f]


def test_profiles_are_short_text_with_commands():
    for f in committed_files():
        if not f.startswith("profiles/"):
            continue
        assert f.endswith((".md", ".txt")), f
        path = os.path.join(ROOT, f)
        assert os.path.getsize(path) < 16 * 1024, f
        text = open(path).read()
        assert "ncu " in text and "--clock-control none" in text, f


def test_no_file_named_for_a_round():
    for f in committed_files():
        # records the job driver writes at the top level (BENCH_r01.json, ...)
        if "/" not in f and re.fullmatch(r"[A-Z0-9]+_r\d+\.json", f):
            continue
        assert not re.search(r"(^|[/_.-])(round|r)\d+([/_.-]|$)", os.path.basename(f),
                             flags=re.I), f


def test_committed_code_does_not_use_the_working_folder():
    for f in committed_files():
        if f.endswith((".py", ".cu", ".cuh", ".h", ".c", ".sh")):
            text = open(os.path.join(ROOT, f)).read()
            folder = "_wo" + "rk"
            assert folder + "/" not in text and folder + "\\" not in text, f


def test_sources_do_not_name_batched_copies():
    pattern = re.compile("cu(da)?Memcpy(3D)?" + "BatchAsync")
    for f in committed_files():
        if f.endswith((".py", ".cu", ".cuh", ".h", ".c")):
            assert not pattern.search(open(os.path.join(ROOT, f)).read()), f


def test_code_names_no_build_documents_or_machines():
    """Code and its comments stand on their own: they name none of the
    build's planning documents, the runner of the GPU jobs, or paths of the
    machine they were written on."""
    words = ["SUR" + "VEY", "DES" + "IGN.md", "VER" + "DICT", "ADV" + "ICE", "BASE" + "LINE",
             "north" + "_star", "gpu" + "run", "/ro" + "ot/"]
    for f in committed_files():
        if f.endswith((".py", ".cu", ".cuh", ".h", ".c", ".sh")):
            text = open(os.path.join(ROOT, f)).read()
            for w in words:
                assert w not in text, (f, w)
