"""Acceptance length of Traversal Verification against token-level
verification on synthetic draft trees (the comparison of §4: Tables 2-4 and
Fig. 4 measure the mean accepted length tau + 1 per cycle for the two
methods on real models; here the same comparison runs on the synthetic
workloads of workloads/synth.py, so only its shape is comparable).

Both methods see the same trees, logits, draft probabilities and uniforms in
every cell; the gain is the paired relative difference of the means.

    python -m workloads.acceptance_study [--batch 512] [--seeds 2] [--vocab 32000]

Prints one markdown table (needs a GPU and the built library).
"""

import argparse
import math

import torch

from workloads.synth import Workload, make_inputs

# tree shapes of §4.1 at depth 5 (chain, binary tree) and the EAGLE-shaped
# sparse tree of the benchmark workloads (depth 6)
SHAPES = {
    "chain, depth 5": ((1, 1, 1, 1, 1), (1, 1, 1, 1, 1)),
    "binary, depth 5": ((2, 4, 8, 16, 32), (2, 2, 2, 2, 2)),
    "EAGLE-shaped, 60 nodes": ((4, 10, 16, 16, 8, 6), (4, 3, 2, 2, 1, 1)),
}
TEMPERATURES = (0.2, 0.4, 0.6, 0.8, 1.0)   # Table 4's range


def cell(tv, levels, branching, vocab, batch, temperature, sigma, seeds):
    """Mean tau + 1 of both methods and the paired relative gain, with the
    standard error of each mean over the valid trees of all seeds.  At low
    temperature a drafted sibling can have draft probability 0 in float32;
    such trees are invalid (tau = -1) for both methods and left out."""
    taus = {"traversal": [], "token": []}
    invalid = 0
    for seed in range(seeds):
        w = Workload("study", batch, vocab, levels, branching, logit_dtype=torch.bfloat16,
                     temperature=temperature, sigma=sigma)
        inp = make_inputs(w, seed=seed, device="cuda")
        got = {}
        for method in taus:
            v = tv.Verifier(vocab, w.nodes, batch, "bf16", method=method)
            _, tau, _ = v.verify(inp.parents, inp.tokens, inp.logits, inp.draft_probs,
                                 inp.temperature, inp.uniforms)
            torch.cuda.synchronize()
            status = v.status()
            v.close()
            if status & ~(tv.TV_STATUS["DEGENERATE"] | tv.TV_STATUS["ZERO_DRAFT"]):
                raise RuntimeError(f"status {status:#x} for {method}")
            got[method] = tau.cpu()
        valid = (got["traversal"] >= 0) & (got["token"] >= 0)
        invalid += int((~valid).sum())
        for method in taus:
            taus[method].append(got[method][valid].double() + 1.0)
        del inp
    out = {}
    for method, ts in taus.items():
        t = torch.cat(ts)
        out[method] = (t.mean().item(), t.std().item() / math.sqrt(t.numel()))
    gain = out["traversal"][0] / out["token"][0] - 1.0
    return out, gain, invalid


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--batch", type=int, default=512)
    ap.add_argument("--seeds", type=int, default=2)
    ap.add_argument("--vocab", type=int, default=32000)
    ap.add_argument("--sigma", type=float, default=1.0)
    args = ap.parse_args()
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    print(f"Mean accepted length tau + 1 (± standard error), V={args.vocab}, bf16 logits, "
          f"draft noise sigma={args.sigma}, {args.batch * args.seeds} trees per cell\n")
    print("| tree | T | token-level | Traversal | gain | invalid trees |")
    print("|---|---|---|---|---|---|")
    for name, (levels, branching) in SHAPES.items():
        for T in TEMPERATURES:
            res, gain, bad = cell(tv, levels, branching, args.vocab, args.batch, T,
                                  args.sigma, args.seeds)
            (mt, st), (mv, sv) = res["token"], res["traversal"]
            print(f"| {name} | {T:.1f} | {mt:.3f} ± {st:.3f} | {mv:.3f} ± {sv:.3f} | "
                  f"{100 * gain:+.1f} % | {bad} |", flush=True)


if __name__ == "__main__":
    main()
