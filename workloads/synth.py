"""Seeded synthetic verification workloads shaped like the paper's.

An input generator only: it draws target logits, draft probabilities, draft
trees and uniforms; no verification arithmetic lives here.

The paper's workloads (Spec-Bench prompts with Llama-3 / Llama-2 / Vicuna
models, §4.1) are not available, so these inputs stand in for them with the
paper's shapes: vocabularies of 32000 (Llama-2 / Vicuna) and 128256
(Llama-3), plus 151936; chain, binary and EAGLE-like sparse trees of depth
5-8 (§4.1, Fig. 4); temperatures in [0.2, 1] (Table 4).

Recipe (all draws seeded, on any torch device):

* target logits  l[b, i, v] = 3 z - 1.1 ln(1 + pi(v)),  z ~ N(0, 1) i.i.d.,
  pi one random permutation of the vocabulary per (workload, seed) shared by
  every row (a Zipf(1.1) rank prior), cast to the logit dtype;
* draft probabilities  q[b, i] = softmax((float(l[b, i]) + sigma n) / T),
  n ~ N(0, 1) i.i.d., float32 -- so sigma sets how far the drafter is from
  the target and hence the acceptance rate;
* workloads: EAGLE-shaped and sweep trees of depth 5-8, and deep768, a
  Sequoia-scale tree of 768 nodes and depth 24; make_inputs_random_shapes
  gives a batch of trees that all differ in shape;
* tree shape from per-level sizes and maximum branching, parents allotted
  greedily to the earliest nodes of the previous level (nodes numbered level
  by level, so parents precede children and the first chain is the deepest);
* the children of every internal node drawn from its draft row without
  replacement, in child-index order (Definition 1), by Gumbel-top-k on
  log q (the sorted top-k of log q + Gumbel noise is distributed as
  sequential sampling without replacement);
* uniforms [B, N+2] ~ U[0, 1) float32;
* for the LM-head pipeline (make_lmhead_inputs): hidden states H [B (N+1), K]
  and an output embedding W [V, K], bf16, with H[:, 0] = 1 and
  W[v, 0] = -1.1 ln(1 + pi(v)) (the same rank prior, as a bias column) and
  the rest N(0, 1) and N(0, 9 / (K - 1)), so l = H W^T has the same law as
  the logits above up to bf16 rounding of the operands; the draft side is
  drawn from those logits as above.
"""

from dataclasses import dataclass, field

import torch


@dataclass
class Workload:
    name: str
    batch: int
    vocab: int
    levels: tuple = ()
    branching: tuple = ()
    parents: tuple = ()
    logit_dtype: torch.dtype = torch.bfloat16
    temperature: float = 1.0
    sigma: float = 1.0
    description: str = ""

    def tree(self):
        if self.parents:
            return list(self.parents)
        return tree_from_levels(self.levels, self.branching)

    @property
    def nodes(self):
        return len(self.tree()) - 1


def tree_from_levels(levels, branching):
    """Parent array (row 0 = root) of a tree with the given per-level sizes,
    each node of a level taking at most ``branching[level]`` children, parents
    allotted greedily to the earliest nodes of the previous level."""
    parents = [-1]
    prev = [0]
    for size, k in zip(levels, branching):
        if size > len(prev) * k:
            raise ValueError("level too large for the branching factor")
        cur = []
        for j in range(size):
            parents.append(prev[j // k])
            cur.append(len(parents) - 1)
        prev = cur
    return parents


EAGLE_LEVELS = (4, 10, 16, 16, 8, 6)
EAGLE_BRANCHING = (4, 3, 2, 2, 1, 1)
# a Sequoia-scale tree (the large, deep trees §4.2 expects larger gains on):
# 768 draft nodes, depth 24, wide near the root and a long tail of chains
DEEP768_LEVELS = (4, 8, 16, 32, 48, 64, 64, 64, 64, 64, 64, 56, 40, 32, 28, 24, 20, 16, 16,
                  12, 12, 8, 8, 4)
DEEP768_BRANCHING = (4, 2, 2, 2, 2, 2) + (1,) * 18

WORKLOADS = {
    "tiny": Workload("tiny", 1, 64, parents=(-1, 0, 0, 1, 1, 2, 2, 3),
                     logit_dtype=torch.float32,
                     description="1 tree, 7 draft nodes, V=64, fp32 logits"),
    "chain8": Workload("chain8", 16, 32000, levels=(1,) * 8, branching=(1,) * 8,
                       logit_dtype=torch.float32,
                       description="16 chains of 8 draft tokens, V=32000, fp32"),
    "binary4": Workload("binary4", 16, 32000, levels=(2, 4, 8, 16),
                        branching=(2, 2, 2, 2), logit_dtype=torch.float32,
                        description="16 binary trees of depth 4 (31 rows), V=32000, fp32"),
    "eagle_v32k": Workload("eagle_v32k", 64, 32000, EAGLE_LEVELS, EAGLE_BRANCHING,
                           description="64 EAGLE-shaped trees (60 nodes, depth 6), V=32000, bf16"),
    "eagle_v128k": Workload("eagle_v128k", 128, 128256, EAGLE_LEVELS, EAGLE_BRANCHING,
                            temperature=0.7,
                            description="128 EAGLE-shaped trees (60 nodes, depth 6), "
                                        "V=128256, bf16, T=0.7"),
    "sweep26": Workload("sweep26", 256, 151936, (2, 4, 8, 8, 4), (2, 2, 2, 1, 1),
                        description="26-node trees, depth 5, V=151936, bf16"),
    "sweep60": Workload("sweep60", 256, 151936, EAGLE_LEVELS, EAGLE_BRANCHING,
                        description="60-node trees, depth 6, V=151936, bf16"),
    "deep768": Workload("deep768", 64, 32000, DEEP768_LEVELS, DEEP768_BRANCHING,
                        description="64 Sequoia-scale trees (768 nodes, depth 24), V=32000, bf16"),
    "sweep120": Workload("sweep120", 256, 151936, (4, 12, 24, 24, 20, 16, 12, 8),
                         (4, 3, 2, 1, 1, 1, 1, 1),
                         description="120-node trees, depth 8, V=151936, bf16"),
}


def get_workload(name, **overrides):
    w = WORKLOADS[name]
    if overrides:
        w = Workload(**{**w.__dict__, **{k: v for k, v in overrides.items() if v is not None}})
    return w


@dataclass
class Inputs:
    parents: torch.Tensor       # [B, N+1] int32
    tokens: torch.Tensor        # [B, N+1] int32
    logits: torch.Tensor        # [B, N+1, V] bf16 / fp32
    draft_probs: torch.Tensor   # [B, N+1, V] fp32
    uniforms: torch.Tensor      # [B, N+2] fp32
    temperature: float
    meta: dict = field(default_factory=dict)


def make_inputs(w: Workload, seed: int = 0, device="cpu", chunk_rows: int = 1 << 14):
    """Draw one batch of the workload on ``device``."""
    dev = torch.device(device)
    parents = w.tree()
    n = len(parents)
    B, V = w.batch, w.vocab
    g = torch.Generator(device=dev).manual_seed(seed)
    perm = torch.randperm(V, generator=g, device=dev)
    bias = -1.1 * torch.log1p(perm.to(torch.float32))
    logits = torch.empty(B, n, V, dtype=w.logit_dtype, device=dev)
    drafts = torch.empty(B, n, V, dtype=torch.float32, device=dev)
    lf = logits.view(B * n, V)
    df = drafts.view(B * n, V)
    rows = B * n
    step = max(1, min(rows, chunk_rows * 1024 // max(V, 1)))
    inv_t = 1.0 / float(w.temperature)
    for r0 in range(0, rows, step):
        r1 = min(rows, r0 + step)
        z = torch.randn(r1 - r0, V, generator=g, device=dev)
        lrow = (3.0 * z + bias).to(w.logit_dtype)
        lf[r0:r1] = lrow
        noise = torch.randn(r1 - r0, V, generator=g, device=dev)
        df[r0:r1] = torch.softmax((lrow.to(torch.float32) + w.sigma * noise) * inv_t, dim=-1)
        del z, noise, lrow

    # children drawn without replacement from the parent's draft row
    gk = torch.Generator(device=dev).manual_seed(seed + 1000)
    tokens = torch.zeros(B, n, dtype=torch.int64, device=dev)
    kids = [[] for _ in range(n)]
    for i in range(1, n):
        kids[parents[i]].append(i)
    for i in range(n):
        if not kids[i]:
            continue
        k = len(kids[i])
        u = torch.rand(B, V, generator=gk, device=dev).clamp_(min=1e-12)
        keys = torch.log(drafts[:, i, :].clamp(min=1e-38)) - torch.log(-torch.log(u))
        top = torch.topk(keys, k, dim=-1, sorted=True).indices
        tokens[:, kids[i]] = top
        del u, keys

    gu = torch.Generator(device=dev).manual_seed(seed + 2000)
    # [B, N+2]: column i tests node i (1..N), column N+1 draws the bonus token
    uniforms = torch.rand(B, n + 1, generator=gu, device=dev)
    uniforms[:, 0] = 0.0
    par = torch.tensor(parents, dtype=torch.int32, device=dev).expand(B, n).contiguous()
    return Inputs(par, tokens.to(torch.int32).contiguous(), logits, drafts,
                  uniforms.contiguous(), float(w.temperature),
                  {"workload": w.name, "seed": seed})


def internal_rows(parents):
    """Indices of rows that have at least one child."""
    has = [False] * len(parents)
    for i in range(1, len(parents)):
        has[parents[i]] = True
    return [i for i, h in enumerate(has) if h]


def random_parents(nodes, rng, width):
    """Parent array (row 0 = root) of a random tree with `nodes` draft nodes:
    node i's parent is drawn uniformly from the `width` nodes before it, so
    small widths give deep, chain-like trees and large ones bushy trees."""
    parents = [-1]
    for i in range(1, nodes + 1):
        parents.append(int(rng.integers(max(0, i - width), i)))
    return parents


def make_inputs_random_shapes(batch, nodes, vocab, seed=0, device="cpu",
                              logit_dtype=torch.bfloat16, temperature=1.0, sigma=1.0,
                              widths=(2, 4, 8, 32)):
    """A batch whose trees all have different random shapes with the same
    node count (tree b uses width widths[b % len(widths)] in random_parents);
    rows, draft probabilities and uniforms as in make_inputs, children drawn
    from their parent's draft row without replacement."""
    import numpy as np
    w = Workload("random_shapes", batch, vocab, parents=tuple([-1] + list(range(nodes))),
                 logit_dtype=logit_dtype, temperature=temperature, sigma=sigma)
    inp = make_inputs(w, seed=seed, device=device)
    dev = inp.logits.device
    rng = np.random.default_rng(seed + 3000)
    shapes = [random_parents(nodes, rng, widths[b % len(widths)]) for b in range(batch)]
    gk = torch.Generator(device=dev).manual_seed(seed + 4000)
    tokens = torch.zeros(batch, nodes + 1, dtype=torch.int64, device=dev)
    for b, parents in enumerate(shapes):
        kids = [[] for _ in range(nodes + 1)]
        for i in range(1, nodes + 1):
            kids[parents[i]].append(i)
        for i, ks in enumerate(kids):
            if not ks:
                continue
            u = torch.rand(vocab, generator=gk, device=dev).clamp_(min=1e-12)
            keys = torch.log(inp.draft_probs[b, i].clamp(min=1e-38)) - torch.log(-torch.log(u))
            tokens[b, ks] = torch.topk(keys, len(ks), sorted=True).indices
    inp.parents = torch.tensor(shapes, dtype=torch.int32, device=dev)
    inp.tokens = tokens.to(torch.int32).contiguous()
    inp.meta = {"workload": f"random_shapes_n{nodes}", "seed": seed}
    return inp


@dataclass
class LmHeadInputs:
    hidden: torch.Tensor        # [B*(N+1), K] bf16
    weight: torch.Tensor        # [V, K] bf16
    inputs: Inputs              # tree, tokens, draft probs, uniforms; logits = bf16(H W^T)


def make_lmhead_inputs(w: Workload, hidden: int = 4096, seed: int = 0, device="cpu",
                       chunk_rows: int = 1 << 14):
    """Hidden states and output embedding whose product is the workload's
    target logits (see the module docstring), plus the draft side drawn from
    those logits.  ``inputs.logits`` holds bf16(H W^T) computed here."""
    dev = torch.device(device)
    parents = w.tree()
    n = len(parents)
    B, V, K = w.batch, w.vocab, hidden
    g = torch.Generator(device=dev).manual_seed(seed)
    perm = torch.randperm(V, generator=g, device=dev)
    H = torch.randn(B * n, K, generator=g, device=dev)
    H[:, 0] = 1.0
    H = H.to(torch.bfloat16)
    W = torch.empty(V, K, dtype=torch.bfloat16, device=dev)
    scale = 3.0 / float(K - 1) ** 0.5
    step = max(1, (chunk_rows * 1024) // K)
    for v0 in range(0, V, step):
        v1 = min(V, v0 + step)
        blk = torch.randn(v1 - v0, K, generator=g, device=dev) * scale
        blk[:, 0] = -1.1 * torch.log1p(perm[v0:v1].to(torch.float32))
        W[v0:v1] = blk.to(torch.bfloat16)
        del blk
    logits = torch.empty(B, n, V, dtype=torch.bfloat16, device=dev)
    lf = logits.view(B * n, V)
    rstep = max(1, (chunk_rows * 1024) // V)
    for r0 in range(0, B * n, rstep):
        r1 = min(B * n, r0 + rstep)
        lf[r0:r1] = (H[r0:r1].float() @ W.float().T if dev.type == "cpu"
                     else H[r0:r1] @ W.T).to(torch.bfloat16)
    inp = _draft_side(w, parents, logits, seed, dev, chunk_rows)
    return LmHeadInputs(H.contiguous(), W.contiguous(), inp)


def _draft_side(w, parents, logits, seed, dev, chunk_rows):
    """Draft probabilities, children and uniforms for given target logits
    (the same recipe as make_inputs)."""
    n = len(parents)
    B, V = w.batch, w.vocab
    g = torch.Generator(device=dev).manual_seed(seed + 500)
    drafts = torch.empty(B, n, V, dtype=torch.float32, device=dev)
    lf = logits.view(B * n, V)
    df = drafts.view(B * n, V)
    step = max(1, min(B * n, chunk_rows * 1024 // max(V, 1)))
    inv_t = 1.0 / float(w.temperature)
    for r0 in range(0, B * n, step):
        r1 = min(B * n, r0 + step)
        noise = torch.randn(r1 - r0, V, generator=g, device=dev)
        df[r0:r1] = torch.softmax((lf[r0:r1].to(torch.float32) + w.sigma * noise) * inv_t,
                                  dim=-1)
        del noise
    gk = torch.Generator(device=dev).manual_seed(seed + 1000)
    tokens = torch.zeros(B, n, dtype=torch.int64, device=dev)
    kids = [[] for _ in range(n)]
    for i in range(1, n):
        kids[parents[i]].append(i)
    for i in range(n):
        if not kids[i]:
            continue
        u = torch.rand(B, V, generator=gk, device=dev).clamp_(min=1e-12)
        keys = torch.log(drafts[:, i, :].clamp(min=1e-38)) - torch.log(-torch.log(u))
        tokens[:, kids[i]] = torch.topk(keys, len(kids[i]), dim=-1, sorted=True).indices
        del u, keys
    gu = torch.Generator(device=dev).manual_seed(seed + 2000)
    uniforms = torch.rand(B, n + 1, generator=gu, device=dev)
    uniforms[:, 0] = 0.0
    par = torch.tensor(parents, dtype=torch.int32, device=dev).expand(B, n).contiguous()
    return Inputs(par, tokens.to(torch.int32).contiguous(), logits, drafts,
                  uniforms.contiguous(), float(w.temperature),
                  {"workload": w.name, "seed": seed, "pipeline": "lmhead"})
