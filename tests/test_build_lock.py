"""Concurrent builds (e.g. every rank of a multi-GPU run calling build())
are serialised: the build lock is held by one process at a time."""

import multiprocessing as mp
import time


def _hold(path):
    from paper_2505_12398_gb300.build import with_build_lock

    def fn():
        t0 = time.time()
        time.sleep(0.4)
        with open(path, "a") as f:
            f.write(f"{t0} {time.time()}\n")

    with_build_lock(fn)


def test_build_lock_serialises_processes(tmp_path):
    out = tmp_path / "intervals"
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_hold, args=(str(out),)) for _ in range(3)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    spans = sorted(tuple(map(float, line.split())) for line in out.read_text().splitlines())
    assert len(spans) == 3
    for (_, end), (start, _) in zip(spans, spans[1:]):
        assert start >= end
