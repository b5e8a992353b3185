#!/usr/bin/env python3
"""Benchmark of batched Traversal Verification (arXiv 2505.12398) on GB300.

One step = one call of the library's verification (tv_verify_batch) over one
batch of synthetic draft trees whose inputs are resident in HBM: the row
normalisers the traversal needs, the serial leaf-to-root traversal of every
tree with its vocabulary-wide rejection passes, and the bonus-token draw.  L2 is flushed (a 256 MiB write) before every timed step, outside the
timed interval.  Times are CUDA-event device times on the launching stream.

Prints ONE JSON line (rank 0).  ``--impl reference`` times the CPU oracle
(the slow literal float64 restatement of the paper's algorithm) on the host
cores instead, on a bounded sample of the same workload per step.

``--pipeline`` times the steps on either side of the verification as well:
``draft`` (drawing every node's children without replacement, Definition 1),
``lmhead`` (the target's logits and row normalisers on the tensor cores, then
verification with them) and ``full`` (drafting, LM head, verification).
"""

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

# The headline: the largest single-GPU throughput configuration, 60-node
# EAGLE-shaped trees at V = 151936 (bf16), 1024 trees, draft noise 2 (the
# low-acceptance end of the sweep).  The other pipelines default to the
# 128-tree, V = 128256 workload.
DEFAULT_VERIFY = ("sweep60", 1024, 2.0)
DEFAULT_WORKLOAD = "eagle_v128k"


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=None)
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--sigma", type=float, default=None)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--method", choices=["traversal", "token"], default="traversal",
                    help="verification method: Traversal Verification, or the token-level "
                         "(top-down RRS without replacement) verifier it is compared with")
    ap.add_argument("--path", choices=["auto", "persistent", "cluster", "three"], default="auto",
                    help="kernel path of the handle (auto: the library's choice)")
    ap.add_argument("--pipeline", choices=["verify", "lmhead", "draft", "full"],
                    default="verify",
                    help="verify: one step = one verification call; lmhead: one step = the "
                         "target LM head (logits and row normalisers on the tensor cores) "
                         "followed by verification with those normalisers; draft: one step = "
                         "drafting every node's children without replacement; full: drafting, "
                         "then the LM head, then verification")
    ap.add_argument("--hidden", type=int, default=4096,
                    help="hidden size K of the LM head (--pipeline lmhead)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="rough budget of the CPU-baseline sample")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the other workloads timed after the headline one")
    ap.add_argument("--extra-steps", type=int, default=20)
    args = ap.parse_args()
    if args.workload is None:
        if args.pipeline == "verify":
            args.workload = DEFAULT_VERIFY[0]
            args.batch = DEFAULT_VERIFY[1] if args.batch is None else args.batch
            args.sigma = DEFAULT_VERIFY[2] if args.sigma is None else args.sigma
        else:
            args.workload = DEFAULT_WORKLOAD
    return args


# ------------------------------------------------------ multi-rank ---------
#
# Trees are independent, so N ranks (one GPU each) verify N batches of their
# own (weak scaling, no collective on the data path).  The only exchanges are
# the barriers around the timed region and the max-reduction of its length.

def rank_seed(seed, rank):
    """Input seed of a rank: every rank draws a different batch."""
    return seed + 7919 * rank


def max_over_ranks(value, world, device):
    """The largest of the ranks' values (the slowest rank sets the job time)."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank, world, repeats, total_ms):
    """Units verified by all ranks per second, over `repeats` timed calls."""
    return units_per_rank * world * repeats / (total_ms / 1e3)


# sources of the persistent kernel, in the order its profile's hash covers them
FLOW_SOURCES = ["tv_control.cuh", "tv_device.cuh", "tv_flow.cu", "tv_launch.h", "tv_ptx.cuh"]
GEMM_SOURCES = ["tv_device.cuh", "tv_gemm.cu", "tv_ptx.cuh"]
DRAFT_SOURCES = ["tv_draft.cu"]


def kernel_sources_sha256(kind="persistent", root=None):
    """SHA-256 over name + bytes of the sources of the dominant kernel (kind
    "persistent": the verification kernel; "lmhead": the LM-head GEMM;
    "draft": drafting), the key a committed ncu summary is tied to."""
    import hashlib
    sources = {"lmhead": GEMM_SOURCES, "draft": DRAFT_SOURCES}.get(kind, FLOW_SOURCES)
    h = hashlib.sha256()
    csrc = os.path.join(root or ROOT, "paper_2505_12398_gb300", "csrc")
    for name in sources:
        h.update(name.encode())
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def kernel_traffic(workload, batch, kind="persistent"):
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary of this workload, or None when there is none or the kernel's
    sources have changed since it was taken."""
    path = os.path.join(ROOT, "profiles", f"launches_{workload}_B{batch}_{kind}.md")
    if not os.path.exists(path):
        return None
    fields = {}
    with open(path) as f:
        for line in f:
            key, sep, val = line.strip().partition(":")
            if sep and key in ("kernel-sources-sha256", "dram-bytes-per-launch"):
                fields[key] = val.strip()
    if len(fields) != 2:
        return None
    if kernel_sources_sha256(kind) != fields["kernel-sources-sha256"]:
        return None
    return int(fields["dram-bytes-per-launch"])


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def measured_bf16_peak():
    """Dense bf16 tensor peak in TFLOP/s: the measured burst figure (a kernel
    timed on its own) or the fallback."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


# ----------------------------------------------------------- clocks ---------

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu_index = gpu_index
        self.proc = None
        self.file = None

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50", "-i", str(self.gpu_index)],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [r.split(",") for r in self.file.read().strip().splitlines() if r.strip()]
        os.unlink(self.file.name)
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax = float(r[2])
            except ValueError:
                continue
            for k, name in enumerate(names):
                if r[5 + k].lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------- CPU oracle ---------

def dump_sample(inp, trees, tmpdir):
    """Host copies of a sample of trees (float32 logits) for the oracle."""
    import numpy as np
    idx = list(trees)
    path = os.path.join(tmpdir, "sample.npz")
    np.savez(path, parents=inp.parents[idx].cpu().numpy(), tokens=inp.tokens[idx].cpu().numpy(),
             logits=inp.logits[idx].float().cpu().numpy(),
             drafts=inp.draft_probs[idx].cpu().numpy(), uniforms=inp.uniforms[idx].cpu().numpy())
    # npz members cannot be memory-mapped; expand to a directory of .npy files
    d = np.load(path)
    outdir = os.path.join(tmpdir, "sample")
    os.makedirs(outdir, exist_ok=True)
    for k in d.files:
        np.save(os.path.join(outdir, k + ".npy"), d[k])
    os.unlink(path)
    return outdir


class _DirArrays:
    def __init__(self, path):
        import numpy as np
        self.d = {k[:-4]: np.load(os.path.join(path, k), mmap_mode="r")
                  for k in os.listdir(path) if k.endswith(".npy")}

    def __getitem__(self, k):
        return self.d[k]


def _oracle_dir_worker(args):
    path, b, temperature, method = args
    if method == "token":
        from oracle.tokenlevel import verify_tree
    else:
        from oracle.verify import verify_tree
    d = _DirArrays(path)
    r = verify_tree(d["parents"][b], d["tokens"][b], d["logits"][b], d["drafts"][b],
                    temperature, d["uniforms"][b])
    return r["tau"]


def time_oracle(sample_dir, n_trees, temperature, pool, reps=1, method="traversal"):
    jobs = [(sample_dir, b % n_trees, temperature, method) for b in range(n_trees * reps)]
    t0 = time.perf_counter()
    pool.map(_oracle_dir_worker, jobs, chunksize=1)
    return time.perf_counter() - t0, len(jobs)


# ---------------------------------------------------------- helpers ---------

def algorithmic_bytes(stats, tau, parents, V, logit_bytes):
    """Bytes of target logits and draft probabilities per step, three ways,
    from the debug entry point's per-tree counts (stats columns: tests,
    S-passes, distinct nodes with a pass R, bonus from an original leaf,
    rows normalised):

    * ``unique``: every row the call needed, each counted once -- the target
      rows it normalised, the draft rows of the R nodes with passes (their
      target rows are among the normalised ones) and, when the bonus came
      from an original leaf, that leaf's target row.  The roofline's bytes.
    * ``s8d``: the count A = |I| V s_l + R V 4 + [leaf] V s_l under the
      eager initialisation of Algorithm 3 (every internal row normalised).
    * ``reread``: what the passes stream, re-reads included: every S-pass
      reads its target and draft rows again (the residual it sums depends on
      the previous pass), the bonus reads one row (target only at a leaf).
    Invalid trees count nothing."""
    import torch
    valid = (tau >= 0).to(torch.int64)
    norm = stats[:, 4].to(torch.int64) * valid
    passes = stats[:, 1].to(torch.int64) * valid
    R = stats[:, 2].to(torch.int64) * valid
    leaf = stats[:, 3].to(torch.int64) * valid
    par = parents.to(torch.int64)
    n_int = torch.zeros_like(par)
    n_int.scatter_(1, par[:, 1:].clamp(min=0), 1)
    internal = n_int.sum(1) * valid
    lb = logit_bytes
    unique = norm * V * lb + R * V * 4 + leaf * V * lb
    s8d = internal * V * lb + R * V * 4 + leaf * V * lb
    bonus = torch.where(leaf > 0, V * lb, V * (lb + 4)) * valid
    reread = norm * V * lb + passes * V * (lb + 4) + bonus
    n = max(int(valid.sum()), 1)
    return {"unique": int(unique.sum()), "s8d": int(s8d.sum()), "reread": int(reread.sum()),
            "normaliser": int((norm * V * lb).sum()),
            "R_per_tree": float(R.sum()) / n, "passes_per_tree": float(passes.sum()) / n,
            "rows_normalised_per_tree": float(norm.sum()) / n,
            "internal_rows_per_tree": float(internal.sum()) / n,
            "leaf_bonus_frac": float(leaf.sum()) / n}


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if args.pipeline in ("lmhead", "full"):
            return run_reference_lmhead(args, world, rank)
        if args.pipeline == "draft":
            return run_reference_draft(args, world, rank)
        return run_reference(args, world, rank)
    if args.pipeline in ("lmhead", "full"):
        return main_lmhead(args, world, rank, local_rank)
    if args.pipeline == "draft":
        return main_draft(args, world, rank, local_rank)

    import torch
    import torch.distributed as dist
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    from workloads.synth import get_workload, make_inputs

    if world > 1:
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local_rank if world > 1 else 0)
    torch.cuda.set_device(dev)
    build()

    w = get_workload(args.workload, batch=args.batch, sigma=args.sigma)
    inp = make_inputs(w, seed=rank_seed(args.seed, rank), device=dev)
    B, R = inp.parents.shape
    N, V = R - 1, w.vocab
    lb = 2 if inp.logits.dtype == torch.bfloat16 else 4
    v = tv.Verifier(V, N, B, "bf16" if lb == 2 else "fp32", device=dev.index, path=args.path,
                    method=args.method)
    stream = torch.cuda.current_stream(dev)

    # decisions are a deterministic function of the inputs: one instrumented
    # call gives the rows each tree needs (algorithmic bytes) and tau
    _, tau_d, _, _, stats, margin = v.verify(inp.parents, inp.tokens, inp.logits,
                                             inp.draft_probs, inp.temperature, inp.uniforms,
                                             debug=True, margins=True)
    torch.cuda.synchronize(dev)
    ab = algorithmic_bytes(stats, tau_d, inp.parents, V, lb)
    # near-ties as the GPU itself reports them (decision margin below 1e-5)
    near_ties = {"tests": int((margin[:, 0] < 1e-5).sum()),
                 "bonus": int((margin[:, 1] < 1e-5).sum()),
                 "trees": int(((margin[:, 0] < 1e-5) | (margin[:, 1] < 1e-5)).sum()),
                 "invalid_trees": int((tau_d < 0).sum())}
    row_bytes = ab["normaliser"]
    trav_bytes = ab["reread"] - row_bytes
    path_code, cluster, warps, stages = v.launch_shape(B, N)
    a_bytes = ab["unique"]
    mean_tau1 = float(tau_d.float().mean()) + 1.0
    passes_per_tree = ab["passes_per_tree"]

    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    out = (torch.empty(B, N, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev))
    v.set_phase_timing(True)
    for _ in range(args.warmup):
        flush.zero_()
        v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                 inp.uniforms, out=out, stream=stream)
    torch.cuda.synchronize(dev)

    gpu_idx = 0
    cvd = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    if cvd and cvd.split(",")[dev.index].strip().isdigit():
        gpu_idx = int(cvd.split(",")[dev.index])
    sampler = ClockSampler(gpu_idx)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    step_ms, phase = [], []
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.zero_()
        e0[k].record(stream)
        v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                 inp.uniforms, out=out, stream=stream)
        e1[k].record(stream)
        phase.append(v.last_phase_ms())
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - wall0
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    step_ms = [e0[k].elapsed_time(e1[k]) for k in range(args.steps)]
    total_ms = sum(step_ms)
    total_ms_max = max_over_ranks(total_ms, world, dev)
    v.set_phase_timing(False)

    # end to end through the public API from pinned host buffers
    e2e = None
    if not args.no_e2e:
        # pinned host copies made directly (no pageable intermediate: the
        # headline batch holds tens of GB)
        hp = []
        for x in (inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.uniforms):
            h = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
            h.copy_(x)
            hp.append(h)
        hout = (torch.empty(B, N, dtype=torch.int32).pin_memory(),
                torch.empty(B, dtype=torch.int32).pin_memory(),
                torch.empty(B, dtype=torch.int32).pin_memory())
        v.verify_host(hp[0], hp[1], hp[2], hp[3], inp.temperature, hp[4], hout, stream=stream)
        ks = max(1, args.e2e_steps)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)
        x0 = torch.cuda.Event(enable_timing=True)
        x1 = torch.cuda.Event(enable_timing=True)
        x0.record(stream)
        for _ in range(ks):
            v.verify_host(hp[0], hp[1], hp[2], hp[3], inp.temperature, hp[4], hout,
                          stream=stream)
        x1.record(stream)
        torch.cuda.synchronize(dev)
        e_ms = x0.elapsed_time(x1)
        e_ms_max = max_over_ranks(e_ms, world, dev)
        # what the host entry point copied (it skips the draft rows of leaves)
        h2d, d2h = v.last_host_copy_bytes()
        assert torch.equal(hout[1], out[1].cpu()), "host entry point disagrees"
        e2e = {"value": round(whole_job_rate(B, world, ks, e_ms_max), 3), "unit": "trees/s",
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": ks}

    # CPU baseline: the oracle on host cores, bounded sample of the same batch
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(inp, args, B)

    # free the headline batch, then time the other configurations
    v.close()
    del inp, out, flush
    torch.cuda.empty_cache()
    extras = None
    if world == 1 and not args.no_extra and args.method == "traversal":
        extras = [measure_extra(tv, n, b, sg, args, dev) for n, b, sg in EXTRA_CONFIGS
                  if (n, b, sg if sg is not None else get_workload(n).sigma) !=
                  (w.name, B, w.sigma)]

    peak, peak_kind = measured_peaks()
    ph = [sum(p[i] for p in phase) / len(phase) for i in range(3)]
    if path_code == 0:
        names = ["tv_prep_kernel", "tv_row_stats_kernel", "tv_traverse_kernel"]
        kbytes = [0, row_bytes, trav_bytes]
        launches_per_step = 3
    else:
        # one kernel reads every row the traversal needs; the first two
        # phases are empty (their events are recorded back to back)
        single = "tv_tree_kernel" if path_code == 1 else "tv_flow_kernel"
        names = ["-", "-", single]
        kbytes = [0, 0, a_bytes]
        launches_per_step = 1
    dom = max(range(3), key=lambda i: ph[i])
    traffic = (kernel_traffic(w.name, B)
               if path_code == 2 and args.method == "traversal" else None)
    ms_step = total_ms_max / args.steps
    trees_s = whole_job_rate(B, world, args.steps, total_ms_max)
    step_gbs = a_bytes / (ms_step / 1e3) / 1e9
    dom_gbs = kbytes[dom] / (ph[dom] / 1e3) / 1e9 if ph[dom] > 0 else 0.0
    dom_s = ph[dom] / 1e3 if ph[dom] > 0 else float("inf")

    def frac(nbytes):
        return round(nbytes / dom_s / 1e9 / peak, 4)

    roof = {"bound": "hbm", "kernel": names[dom], "achieved": round(dom_gbs, 2),
            "peak": peak, "unit": "GB/s", "frac": round(dom_gbs / peak, 4),
            "peak_kind": peak_kind, "bytes": "unique rows needed, each once",
            "bytes_per_launch": kbytes[dom], "traffic": traffic}
    if path_code != 0:
        roof["frac_reread_inclusive"] = frac(ab["reread"])
        roof["frac_eager_A"] = frac(ab["s8d"])
        if traffic:
            roof["dram_frac"] = frac(traffic)
            roof["traffic_over_unique"] = round(traffic / max(ab["unique"], 1), 4)
    line = {
        "metric": "verified trees/sec and logit GB/s (fraction of HBM peak) at batch B, "
                  "vocab V, 1 GB300",
        "value": round(trees_s, 3),
        "unit": "trees/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 6),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic (seeded logits with Zipf rank prior, noisy-drafter probabilities, "
                "EAGLE-shaped draft trees sampled without replacement)",
        "config": {"workload": w.name, "batch": B, "vocab": V, "nodes": N, "method": args.method,
                   "logit_dtype": "bf16" if lb == 2 else "fp32",
                   "temperature": w.temperature, "sigma": w.sigma, "seed": args.seed,
                   "l2": "flushed by a 256 MiB write before every timed step (untimed)",
                   "parallelism": f"dp{world} (independent trees per GPU)",
                   "kernel_path": ["three-kernel", "cluster-per-tree",
                                   "persistent"][path_code],
                   "ctas_per_tree": cluster, "consumer_warps": warps, "ring_stages": stages},
        "verified_logit_gbps": round(step_gbs, 2),
        "hbm_frac_step": round(step_gbs / peak, 4),
        "bytes_per_step": {"unique": ab["unique"], "eager_A": ab["s8d"],
                           "reread_inclusive": ab["reread"]},
        "per_tree": {k: round(ab[k], 4) for k in ("R_per_tree", "passes_per_tree",
                                                  "rows_normalised_per_tree",
                                                  "internal_rows_per_tree",
                                                  "leaf_bonus_frac")},
        "mean_accept_len_tau_plus_1": round(mean_tau1, 4),
        "near_ties_margin_below_1e-5": near_ties,
        "phase_ms": {names[i]: round(ph[i], 6) for i in range(3) if names[i] != "-"},
        "roofline": roof,
        "roofline_step": {"bound": "hbm", "achieved": round(step_gbs, 2), "peak": peak,
                          "unit": "GB/s", "frac": round(step_gbs / peak, 4)},
        "e2e": e2e,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
        "cpu_baseline": cpu,
        "other_configs": extras,
        "wall_s_timed_region": round(wall, 3),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# The other configurations, timed after the headline one (one GPU, rank 0):
# 64 EAGLE-shaped trees at V = 32000, 128 at V = 128256 (T = 0.7), and the other
# corners of the V = 151936 throughput sweep.
EXTRA_CONFIGS = (("eagle_v32k", 64, None), ("eagle_v128k", 128, None), ("sweep60", 1024, 0.5),
                 ("sweep26", 1024, 2.0), ("sweep120", 1024, 2.0))


def measure_extra(tv, name, batch, sigma, args, dev):
    """Device time of one more workload on a fresh handle: warm-up, then
    args.extra_steps timed calls (L2 flushed before each), with the same byte
    counts as the headline."""
    import torch
    from workloads.synth import get_workload, make_inputs
    w = get_workload(name, batch=batch, sigma=sigma)
    inp = make_inputs(w, seed=args.seed, device=dev)
    B, R = inp.parents.shape
    N, V = R - 1, w.vocab
    lb = 2 if inp.logits.dtype == torch.bfloat16 else 4
    v = tv.Verifier(V, N, B, "bf16" if lb == 2 else "fp32", device=dev.index, path=args.path,
                    method=args.method)
    stream = torch.cuda.current_stream(dev)
    _, tau_d, _, _, stats = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs,
                                     inp.temperature, inp.uniforms, debug=True)
    torch.cuda.synchronize(dev)
    ab = algorithmic_bytes(stats, tau_d, inp.parents, V, lb)
    out = (torch.empty(B, N, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev))
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    times = []
    for k in range(max(3, args.warmup) + args.extra_steps):
        flush.zero_()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs, inp.temperature,
                 inp.uniforms, out=out, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        if k >= max(3, args.warmup):
            times.append(e0.elapsed_time(e1))
    status = v.status()
    v.close()
    del inp, flush, out
    torch.cuda.empty_cache()
    peak, _ = measured_peaks()
    ms = sum(times) / len(times)
    sec = ms / 1e3
    return {"workload": name, "batch": B, "vocab": V, "nodes": N, "sigma": w.sigma,
            "temperature": w.temperature, "steps": len(times), "ms_per_step": round(ms, 6),
            "trees_per_s": round(B / sec, 1),
            "frac_unique": round(ab["unique"] / sec / 1e9 / peak, 4),
            "frac_reread_inclusive": round(ab["reread"] / sec / 1e9 / peak, 4),
            "frac_eager_A": round(ab["s8d"] / sec / 1e9 / peak, 4),
            "bytes_per_step": {"unique": ab["unique"], "eager_A": ab["s8d"],
                               "reread_inclusive": ab["reread"]},
            "per_tree": {k: round(ab[k], 4) for k in ("R_per_tree", "passes_per_tree",
                                                      "rows_normalised_per_tree",
                                                      "internal_rows_per_tree")},
            "status": int(status)}


def cpu_baseline(inp, args, B):
    import multiprocessing as mp
    cores = os.cpu_count() or 1
    with tempfile.TemporaryDirectory() as td:
        n_sample = min(B, max(cores, 8))
        sdir = dump_sample(inp, range(n_sample), td)
        ctx = mp.get_context("spawn")
        with ctx.Pool(cores) as pool:
            # one probe tree per worker to size the sample to the time budget,
            # after an untimed round that starts the workers and loads the arrays
            time_oracle(sdir, n_sample, inp.temperature, pool, method=args.method)
            t_probe, n_probe = time_oracle(sdir, n_sample, inp.temperature, pool,
                                           method=args.method)
            per_round = max(t_probe, 1e-3)
            reps = max(1, min(5000, int(args.cpu_seconds / per_round)))
            t, n = time_oracle(sdir, n_sample, inp.temperature, pool, reps=reps,
                               method=args.method)
    return {"value": round(n / t, 4), "unit": "trees/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} oracle tree verifications ({n_sample} distinct trees of the same "
                      f"batch, repeated {reps}x) across {cores} spawn workers, {t:.1f} s"}


def run_reference(args, world, rank):
    """The oracle (float64 CPU restatement of Algorithm 3) as the reference arm."""
    if rank != 0:
        return
    import multiprocessing as mp
    from workloads.synth import get_workload, make_inputs
    w = get_workload(args.workload, batch=args.batch, sigma=args.sigma)
    cores = os.cpu_count() or 1
    per_step = max(1, min(w.batch, cores))
    # the same workload, drawn on the CPU; only the sampled trees are needed
    gen_w = get_workload(args.workload, batch=per_step, sigma=args.sigma)
    inp = make_inputs(gen_w, seed=args.seed, device="cpu")
    with tempfile.TemporaryDirectory() as td:
        sdir = dump_sample(inp, range(per_step), td)
        ctx = mp.get_context("spawn")
        with ctx.Pool(cores) as pool:
            for _ in range(args.warmup):
                time_oracle(sdir, per_step, inp.temperature, pool, method=args.method)
            times = []
            for _ in range(args.steps):
                t, _ = time_oracle(sdir, per_step, inp.temperature, pool, method=args.method)
                times.append(t)
    total = sum(times)
    value = per_step * args.steps / total
    line = {
        "impl": "reference",
        "metric": "verified trees/sec and logit GB/s (fraction of HBM peak) at batch B, "
                  "vocab V, 1 GB300",
        "value": round(value, 4), "unit": "trees/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": w.name, "batch": w.batch, "vocab": w.vocab,
                                         "method": args.method,
                                         "nodes": w.nodes},
        "cpu_baseline": {"value": round(value, 4), "unit": "trees/s", "cores": cores,
                         "kind": "oracle",
                         "sample": f"{per_step} trees of the workload per step, one per "
                                   f"spawn worker"},
        "e2e": {"value": round(value, 4), "unit": "trees/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------- LM-head pipeline ---------

def dump_lmhead_sample(lin, trees, tmpdir, u_draft=None):
    """Host copies, for the oracle, of the sampled trees' hidden states and
    draft side, and of the output embedding (bf16 bit patterns)."""
    import numpy as np
    import torch
    inp = lin.inputs
    idx = list(trees)
    R = inp.parents.shape[1]
    outdir = os.path.join(tmpdir, "lmhead")
    os.makedirs(outdir, exist_ok=True)
    rows = torch.cat([torch.arange(b * R, (b + 1) * R) for b in idx]).to(lin.hidden.device)
    arrays = {
        "hidden": lin.hidden.index_select(0, rows).view(torch.int16).cpu().numpy(),
        "weight": lin.weight.view(torch.int16).cpu().numpy(),
        "parents": inp.parents[idx].cpu().numpy(), "tokens": inp.tokens[idx].cpu().numpy(),
        "drafts": inp.draft_probs[idx].cpu().numpy(), "uniforms": inp.uniforms[idx].cpu().numpy(),
    }
    if u_draft is not None:
        arrays["udraft"] = u_draft[idx].cpu().numpy()
    for k, a in arrays.items():
        np.save(os.path.join(outdir, k + ".npy"), a)
    return outdir


def _bf16_bits_to_f64(a):
    import numpy as np
    return (a.astype(np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _lmhead_oracle_worker(args):
    """One tree through the oracle: logits of its rows (float64 products,
    stored as bf16), then Algorithm 3 on them."""
    path, b, temperature = args
    import numpy as np
    from oracle import lmhead
    from oracle.verify import verify_tree
    d = _DirArrays(path)
    R = d["parents"].shape[1]
    h = _bf16_bits_to_f64(np.asarray(d["hidden"][b * R:(b + 1) * R]))
    wt = d["weight"]
    V = wt.shape[0]
    logits = np.empty((R, V))
    step = 8192                       # output columns per chunk: bounds the float64 copy of W
    for v0 in range(0, V, step):
        v1 = min(V, v0 + step)
        logits[:, v0:v1] = lmhead.logits(h, _bf16_bits_to_f64(np.asarray(wt[v0:v1])))
    stored = lmhead.to_bf16(logits)
    tokens = d["tokens"][b]
    if "udraft" in d.d:                # the full pipeline drafts the tree first
        from oracle.drafting import sample_tree
        tokens = np.asarray(sample_tree(d["parents"][b], d["drafts"][b],
                                        [float(x) for x in d["udraft"][b]]))
    r = verify_tree(d["parents"][b], tokens, stored, d["drafts"][b], temperature,
                    d["uniforms"][b])
    return r["tau"]


def time_lmhead_oracle(sample_dir, n_trees, temperature, pool, reps=1):
    jobs = [(sample_dir, b % n_trees, temperature) for b in range(n_trees * reps)]
    t0 = time.perf_counter()
    taus = pool.map(_lmhead_oracle_worker, jobs, chunksize=1)
    return time.perf_counter() - t0, len(jobs), taus


def _oracle_pool(cores):
    """A spawn pool whose workers run single-threaded BLAS (one tree each)."""
    import multiprocessing as mp
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[k] = "1"
    return mp.get_context("spawn").Pool(cores)


LMHEAD_METRIC = {
    "lmhead": "verified trees/sec including the target LM head (logits + row normalisers on "
              "the tensor cores, then verification), 1 GB300",
    "full": "drafted and verified trees/sec (drafting without replacement, the target LM "
            "head with its row normalisers, then verification), 1 GB300",
}


def main_lmhead(args, world, rank, local_rank):
    """One step = tv_lm_head (logits and row normalisers of every row of the
    batch, tensor cores) then tv_verify_batch_stats on them; with --pipeline
    full, tv_draft_children first draws the trees' tokens."""
    import torch
    import torch.distributed as dist
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    from workloads.synth import get_workload, make_lmhead_inputs

    if world > 1:
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local_rank if world > 1 else 0)
    torch.cuda.set_device(dev)
    build()

    w = get_workload(args.workload, batch=args.batch, sigma=args.sigma,
                     logit_dtype=torch.bfloat16)
    lin = make_lmhead_inputs(w, hidden=args.hidden, seed=rank_seed(args.seed, rank), device=dev)
    inp = lin.inputs
    B, R = inp.parents.shape
    N, V, K = R - 1, w.vocab, args.hidden
    M = B * R
    v = tv.Verifier(V, N, B, "bf16", device=dev.index, path="persistent", method=args.method)
    stream = torch.cuda.current_stream(dev)
    logits = torch.empty(B, R, V, dtype=torch.bfloat16, device=dev)
    row_stats = torch.empty(M, 2, dtype=torch.float32, device=dev)
    lm_out = (logits.view(M, V), row_stats)
    out = (torch.empty(B, N, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev))
    full = args.pipeline == "full"
    gd = torch.Generator(device=dev).manual_seed(rank_seed(args.seed, rank) + 3000)
    u_draft = torch.rand(B, R, generator=gd, device=dev)
    tokens = torch.empty(B, R, dtype=torch.int32, device=dev)
    # the per-step input besides hidden states and the draft side: the drafting
    # uniforms (full pipeline) or the draft tokens
    side0 = u_draft if full else inp.tokens

    def step(ev=None, hidden=lin.hidden, parents=inp.parents, drafts=inp.draft_probs,
             uniforms=inp.uniforms, side=side0, debug=False):
        toks = side
        if full:
            v.draft_children(parents, drafts, side, out=tokens, stream=stream)
            toks = tokens
        if ev is not None:
            ev[1].record(stream)
        v.lm_head(hidden, lin.weight, inp.temperature, out=lm_out, stream=stream)
        if ev is not None:
            ev[2].record(stream)
        return v.verify_stats(parents, toks, logits, drafts, inp.temperature, uniforms,
                              row_stats, out=None if debug else out, stream=stream, debug=debug)

    # instrumented call: the rows each tree reads, tau
    _, tau_d, _, _, stats = step(debug=True)
    torch.cuda.synchronize(dev)
    if v.status() & ~16:
        raise RuntimeError(f"device status {tv.status_names(v.status())}")
    ab = algorithmic_bytes(stats, tau_d, inp.parents, V, 2)
    trav_bytes = ab["reread"] - ab["normaliser"]
    mean_tau1 = float(tau_d.float().mean()) + 1.0

    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        flush.zero_()
        step()
    torch.cuda.synchronize(dev)

    gpu_idx = 0
    cvd = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    if cvd and cvd.split(",")[dev.index].strip().isdigit():
        gpu_idx = int(cvd.split(",")[dev.index])
    sampler = ClockSampler(gpu_idx)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.zero_()
        ev[k][0].record(stream)
        step(ev[k])
        ev[k][3].record(stream)
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - wall0
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    draft_ms = sum(e[0].elapsed_time(e[1]) for e in ev) / args.steps
    gemm_ms = sum(e[1].elapsed_time(e[2]) for e in ev) / args.steps
    ver_ms = sum(e[2].elapsed_time(e[3]) for e in ev) / args.steps
    total_ms = sum(e[0].elapsed_time(e[3]) for e in ev)
    total_ms_max = max_over_ranks(total_ms, world, dev)

    # end to end: hidden states and the draft side from pinned host memory,
    # outputs back to the host, every step
    e2e = None
    if not args.no_e2e:
        hp = [x.cpu().pin_memory() for x in (lin.hidden, inp.parents, side0,
                                              inp.draft_probs, inp.uniforms)]
        dbuf = [torch.empty_like(x, device=dev) for x in hp]
        hout = [torch.empty(o.shape, dtype=o.dtype).pin_memory() for o in out]

        def e2e_step():
            for d, h in zip(dbuf, hp):
                d.copy_(h, non_blocking=True)
            step(hidden=dbuf[0], parents=dbuf[1], side=dbuf[2], drafts=dbuf[3],
                 uniforms=dbuf[4])
            for h, o in zip(hout, out):
                h.copy_(o, non_blocking=True)

        e2e_step()
        torch.cuda.synchronize(dev)
        ks = max(1, args.e2e_steps)
        if world > 1:
            dist.barrier()
        x0 = torch.cuda.Event(enable_timing=True)
        x1 = torch.cuda.Event(enable_timing=True)
        x0.record(stream)
        for _ in range(ks):
            e2e_step()
        x1.record(stream)
        torch.cuda.synchronize(dev)
        e_ms_max = max_over_ranks(x0.elapsed_time(x1), world, dev)
        assert torch.equal(hout[1], out[1].cpu()), "end-to-end outputs disagree"
        e2e = {"value": round(whole_job_rate(B, world, ks, e_ms_max), 3), "unit": "trees/s",
               "h2d_bytes_per_step": int(sum(x.numel() * x.element_size() for x in hp)),
               "d2h_bytes_per_step": int(sum(x.numel() * x.element_size() for x in hout)),
               "steps": ks}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_lmhead(lin, args, B, u_draft if full else None)

    peak, peak_kind = measured_bf16_peak()
    hbm, hbm_kind = measured_peaks()
    flops = 2.0 * M * K * V
    gemm_tflops = flops / (gemm_ms / 1e3) / 1e12
    ver_gbs = trav_bytes / (ver_ms / 1e3) / 1e9
    ms_step = total_ms_max / args.steps
    phases = {"lm_head_kernel+lm_head_merge_kernel": round(gemm_ms, 6),
              "tv_flow_kernel (given normalisers)": round(ver_ms, 6)}
    if full:
        phases = {"tv_draft_kernel": round(draft_ms, 6), **phases}
    line = {
        "metric": LMHEAD_METRIC[args.pipeline],
        "value": round(whole_job_rate(B, world, args.steps, total_ms_max), 3),
        "unit": "trees/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_step, 6), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (hidden states and output embedding whose product has the "
                "workload's logit law; draft side drawn from those logits)",
        "config": {"workload": w.name, "pipeline": args.pipeline, "batch": B, "vocab": V,
                   "nodes": N, "hidden": K, "rows": M, "method": args.method,
                   "temperature": w.temperature, "sigma": w.sigma, "seed": args.seed,
                   "l2": "flushed by a 256 MiB write before every timed step (untimed)",
                   "parallelism": f"dp{world} (independent trees per GPU)"},
        "phase_ms": phases,
        "mean_accept_len_tau_plus_1": round(mean_tau1, 4),
        "roofline": {"bound": "tensor", "kernel": "lm_head_kernel",
                     "achieved": round(gemm_tflops, 2), "peak": peak, "unit": "TFLOP/s",
                     "frac": round(gemm_tflops / peak, 4), "peak_kind": peak_kind + " (burst)",
                     "flops_per_launch": flops,
                     "traffic": kernel_traffic(w.name, B, "lmhead")},
        "roofline_verify": {"bound": "hbm", "kernel": "tv_flow_kernel",
                            "achieved": round(ver_gbs, 2), "peak": hbm, "unit": "GB/s",
                            "frac": round(ver_gbs / hbm, 4), "peak_kind": hbm_kind,
                            "bytes_per_launch": trav_bytes},
        "e2e": e2e,
        "gpu_launches": (4 if full else 3) * args.steps,
        "clocks": clocks,
        "cpu_baseline": cpu,
        "wall_s_timed_region": round(wall, 3),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    v.close()
    if world > 1:
        dist.destroy_process_group()


def cpu_baseline_lmhead(lin, args, B, u_draft=None):
    cores = os.cpu_count() or 1
    with tempfile.TemporaryDirectory() as td:
        n_sample = min(B, cores)
        sdir = dump_lmhead_sample(lin, range(n_sample), td, u_draft)
        with _oracle_pool(cores) as pool:
            t_probe, _, _ = time_lmhead_oracle(sdir, n_sample, lin.inputs.temperature, pool)
            reps = max(1, min(50, int(args.cpu_seconds / max(t_probe, 1e-3))))
            t, n, _ = time_lmhead_oracle(sdir, n_sample, lin.inputs.temperature, pool, reps=reps)
    return {"value": round(n / t, 4), "unit": "trees/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} trees ({n_sample} distinct trees of the batch, repeated {reps}x) "
                      + ("drafted by the oracle, " if u_draft is not None else "")
                      + f"through the oracle LM head (float64 products, bf16 storage) and "
                      f"verification, one tree per single-threaded spawn worker, {t:.1f} s"}


def run_reference_lmhead(args, world, rank):
    """The oracle LM head and verification as the reference arm."""
    if rank != 0:
        return
    import torch
    from workloads.synth import get_workload, make_lmhead_inputs
    w = get_workload(args.workload, batch=args.batch, sigma=args.sigma)
    cores = os.cpu_count() or 1
    per_step = max(1, min(w.batch, cores))
    gen_w = get_workload(args.workload, batch=per_step, sigma=args.sigma,
                         logit_dtype=torch.bfloat16)
    lin = make_lmhead_inputs(gen_w, hidden=args.hidden, seed=args.seed, device="cpu")
    u_draft = None
    if args.pipeline == "full":
        g = torch.Generator().manual_seed(args.seed + 3000)
        u_draft = torch.rand(per_step, lin.inputs.parents.shape[1], generator=g)
    with tempfile.TemporaryDirectory() as td:
        sdir = dump_lmhead_sample(lin, range(per_step), td, u_draft)
        with _oracle_pool(cores) as pool:
            for _ in range(args.warmup):
                time_lmhead_oracle(sdir, per_step, lin.inputs.temperature, pool)
            times = [time_lmhead_oracle(sdir, per_step, lin.inputs.temperature, pool)[0]
                     for _ in range(args.steps)]
    total = sum(times)
    value = per_step * args.steps / total
    line = {
        "impl": "reference",
        "metric": LMHEAD_METRIC[args.pipeline],
        "value": round(value, 4), "unit": "trees/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": w.name, "pipeline": args.pipeline, "batch": w.batch,
                   "vocab": w.vocab, "nodes": w.nodes, "hidden": args.hidden,
                   "method": args.method},
        "cpu_baseline": {"value": round(value, 4), "unit": "trees/s", "cores": cores,
                         "kind": "oracle",
                         "sample": f"{per_step} trees of the workload per step, one per "
                                   f"single-threaded spawn worker"},
        "e2e": {"value": round(value, 4), "unit": "trees/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------- drafting ---------

def _draft_oracle_worker(args):
    path, b = args
    from oracle.drafting import sample_tree
    d = _DirArrays(path)
    return sample_tree(d["parents"][b], d["drafts"][b], [float(x) for x in d["uniforms"][b]])


def main_draft(args, world, rank, local_rank):
    """One step = tv_draft_children over the batch: every node's token drawn
    from its parent's draft row without its earlier siblings' tokens."""
    import numpy as np
    import torch
    import torch.distributed as dist
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    from workloads.synth import get_workload, internal_rows, make_inputs

    if world > 1:
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local_rank if world > 1 else 0)
    torch.cuda.set_device(dev)
    build()
    w = get_workload(args.workload, batch=args.batch, sigma=args.sigma)
    inp = make_inputs(w, seed=rank_seed(args.seed, rank), device=dev)
    B, R = inp.parents.shape
    N, V = R - 1, w.vocab
    g = torch.Generator(device=dev).manual_seed(rank_seed(args.seed, rank) + 3000)
    u = torch.rand(B, R, generator=g, device=dev)
    v = tv.Verifier(V, N, B, "bf16", device=dev.index, path="three")
    stream = torch.cuda.current_stream(dev)
    out = torch.empty(B, R, dtype=torch.int32, device=dev)
    n_int = len(internal_rows(w.tree()))
    a_bytes = B * n_int * V * 4 + B * R * 12      # internal draft rows once; parents, u, tokens

    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        flush.zero_()
        v.draft_children(inp.parents, inp.draft_probs, u, out=out, stream=stream)
    torch.cuda.synchronize(dev)
    if v.status():
        raise RuntimeError(f"device status {tv.status_names(v.status())}")
    gpu_idx = 0
    cvd = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    if cvd and cvd.split(",")[dev.index].strip().isdigit():
        gpu_idx = int(cvd.split(",")[dev.index])
    sampler = ClockSampler(gpu_idx)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.zero_()
        ev[k][0].record(stream)
        v.draft_children(inp.parents, inp.draft_probs, u, out=out, stream=stream)
        ev[k][1].record(stream)
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - wall0
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = sum(e[0].elapsed_time(e[1]) for e in ev)
    total_ms_max = max_over_ranks(total_ms, world, dev)

    e2e = None
    if not args.no_e2e:
        hp = [x.cpu().pin_memory() for x in (inp.parents, inp.draft_probs, u)]
        dbuf = [torch.empty_like(x, device=dev) for x in hp]
        hout = torch.empty(B, R, dtype=torch.int32).pin_memory()

        def e2e_step():
            for d, h in zip(dbuf, hp):
                d.copy_(h, non_blocking=True)
            v.draft_children(dbuf[0], dbuf[1], dbuf[2], out=out, stream=stream)
            hout.copy_(out, non_blocking=True)

        e2e_step()
        torch.cuda.synchronize(dev)
        ks = max(1, args.e2e_steps)
        if world > 1:
            dist.barrier()
        x0 = torch.cuda.Event(enable_timing=True)
        x1 = torch.cuda.Event(enable_timing=True)
        x0.record(stream)
        for _ in range(ks):
            e2e_step()
        x1.record(stream)
        torch.cuda.synchronize(dev)
        e_ms_max = max_over_ranks(x0.elapsed_time(x1), world, dev)
        assert torch.equal(hout, out.cpu()), "end-to-end tokens disagree"
        e2e = {"value": round(whole_job_rate(B, world, ks, e_ms_max), 3), "unit": "trees/s",
               "h2d_bytes_per_step": int(sum(x.numel() * x.element_size() for x in hp)),
               "d2h_bytes_per_step": int(hout.numel() * hout.element_size()), "steps": ks}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cores = os.cpu_count() or 1
        n_sample = min(B, max(cores, 8))
        with tempfile.TemporaryDirectory() as td:
            sdir = os.path.join(td, "draft")
            os.makedirs(sdir)
            for k, a in (("parents", inp.parents[:n_sample]), ("drafts", inp.draft_probs[:n_sample]),
                         ("uniforms", u[:n_sample])):
                np.save(os.path.join(sdir, k + ".npy"), a.cpu().numpy())
            with _oracle_pool(cores) as pool:
                jobs = [(sdir, b) for b in range(n_sample)]
                t0 = time.perf_counter()
                pool.map(_draft_oracle_worker, jobs, chunksize=1)
                t_probe = time.perf_counter() - t0
                reps = max(1, min(200, int(args.cpu_seconds / max(t_probe, 1e-3))))
                t0 = time.perf_counter()
                pool.map(_draft_oracle_worker, jobs * reps, chunksize=1)
                t = time.perf_counter() - t0
        n = n_sample * reps
        cpu = {"value": round(n / t, 4), "unit": "trees/s", "cores": cores, "kind": "oracle",
               "sample": f"{n} trees ({n_sample} distinct trees of the batch, repeated {reps}x) "
                         f"drafted by the oracle, one tree per single-threaded spawn worker, "
                         f"{t:.1f} s"}

    peak, peak_kind = measured_peaks()
    ms_step = total_ms_max / args.steps
    gbs = a_bytes / (ms_step / 1e3) / 1e9
    line = {
        "metric": "drafted trees/sec (every node's children drawn without replacement from "
                  "its draft row, Definition 1) and draft-row GB/s, 1 GB300",
        "value": round(whole_job_rate(B, world, args.steps, total_ms_max), 3),
        "unit": "trees/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_step, 6), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (noisy-drafter probabilities of the workload, uniforms U[0,1))",
        "config": {"workload": w.name, "pipeline": "draft", "batch": B, "vocab": V, "nodes": N,
                   "internal_rows_per_tree": n_int, "seed": args.seed,
                   "l2": "flushed by a 256 MiB write before every timed step (untimed)",
                   "parallelism": f"dp{world} (independent trees per GPU)"},
        "roofline": {"bound": "hbm", "kernel": "tv_draft_kernel", "achieved": round(gbs, 2),
                     "peak": peak, "unit": "GB/s", "frac": round(gbs / peak, 4),
                     "peak_kind": peak_kind, "bytes_per_launch": a_bytes,
                     "traffic": kernel_traffic(w.name, B, "draft")},
        "e2e": e2e, "gpu_launches": args.steps, "clocks": clocks, "cpu_baseline": cpu,
        "wall_s_timed_region": round(wall, 3),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    v.close()
    if world > 1:
        dist.destroy_process_group()


def run_reference_draft(args, world, rank):
    """The drafting oracle as the reference arm."""
    if rank != 0:
        return
    import numpy as np
    import torch
    from workloads.synth import get_workload, make_inputs
    w = get_workload(args.workload, batch=args.batch, sigma=args.sigma)
    cores = os.cpu_count() or 1
    per_step = max(1, min(w.batch, cores))
    inp = make_inputs(get_workload(args.workload, batch=per_step, sigma=args.sigma),
                      seed=args.seed, device="cpu")
    g = torch.Generator().manual_seed(args.seed + 3000)
    u = torch.rand(per_step, inp.parents.shape[1], generator=g)
    with tempfile.TemporaryDirectory() as td:
        for k, a in (("parents", inp.parents), ("drafts", inp.draft_probs), ("uniforms", u)):
            np.save(os.path.join(td, k + ".npy"), a.numpy())
        jobs = [(td, b) for b in range(per_step)]
        with _oracle_pool(cores) as pool:
            for _ in range(args.warmup):
                pool.map(_draft_oracle_worker, jobs, chunksize=1)
            times = []
            for _ in range(args.steps):
                t0 = time.perf_counter()
                pool.map(_draft_oracle_worker, jobs, chunksize=1)
                times.append(time.perf_counter() - t0)
    total = sum(times)
    value = per_step * args.steps / total
    print(json.dumps({
        "impl": "reference",
        "metric": "drafted trees/sec (every node's children drawn without replacement from "
                  "its draft row, Definition 1) and draft-row GB/s, 1 GB300",
        "value": round(value, 4), "unit": "trees/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": w.name, "pipeline": "draft", "batch": w.batch, "vocab": w.vocab,
                   "nodes": w.nodes},
        "cpu_baseline": {"value": round(value, 4), "unit": "trees/s", "cores": cores,
                         "kind": "oracle",
                         "sample": f"{per_step} trees of the workload per step, one per "
                                   f"single-threaded spawn worker"},
        "e2e": {"value": round(value, 4), "unit": "trees/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


if __name__ == "__main__":
    main()
