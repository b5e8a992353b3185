"""CPU checks of the error bounds the GPU parity tests rely on, by replaying
the kernels' own float32 / float64 operation order with numpy (IEEE
round-to-nearest-even in both, as on the GPU).

Drafting (tv_draft.cu): a lane sums its 8 tokens pairwise in float32, a warp
adds its 32 lane sums with a 5-step xor butterfly in float32 (a 256-token
tile sum), and warp 0 turns the tile sums into a float64 inclusive prefix (a
sequential run of tiles per lane, a Hillis-Steele scan of the run totals
across lanes, then the run again).  The GPU drafting tests allow a token to
differ from the oracle's only when u W is within 1e-6 W of a step of the
exact CDF; these tests measure how far the kernel's prefix is from the exact
one."""

import numpy as np
import pytest

TILE = 256


def tile_sums_f32(q):
    """The kernel's float32 tile sums of a row (zeros past the end)."""
    V = len(q)
    n_tiles = (V + TILE - 1) // TILE
    x = np.zeros(n_tiles * TILE, dtype=np.float32)
    x[:V] = q.astype(np.float32)
    v = x.reshape(n_tiles, 32, 8)
    s = ((v[..., 0] + v[..., 1]) + (v[..., 2] + v[..., 3])) + \
        ((v[..., 4] + v[..., 5]) + (v[..., 6] + v[..., 7]))       # [tiles, 32] lane sums
    lane = np.arange(32)
    for o in (16, 8, 4, 2, 1):                                     # xor butterfly
        s = (s + s[:, lane ^ o]).astype(np.float32)
    return s[:, 0]


def prefix_f64(tsum):
    """The kernel's float64 inclusive prefix of the tile sums."""
    n = len(tsum)
    per = (n + 31) // 32
    acc = np.zeros(32)
    for lane in range(32):
        t0, t1 = min(n, lane * per), min(n, lane * per + per)
        a = 0.0
        for t in range(t0, t1):
            a += float(tsum[t])
        acc[lane] = a
    x = acc.copy()
    for o in (1, 2, 4, 8, 16):                                     # Hillis-Steele
        y = np.concatenate([np.zeros(o), x[:-o]])
        x = np.where(np.arange(32) >= o, x + y, x)
    ex = x - acc
    out = np.zeros(n)
    for lane in range(32):
        t0, t1 = min(n, lane * per), min(n, lane * per + per)
        run = ex[lane]
        for t in range(t0, t1):
            run += float(tsum[t])
            out[t] = run
    return out


def test_replay_matches_a_direct_sum_on_exact_rows():
    """On dyadic rows every float32 and float64 sum is exact, so the replay
    must give the exact prefix (a check of the replay itself)."""
    rng = np.random.default_rng(0)
    q = rng.integers(0, 64, 5000).astype(np.float64) / 1024.0
    got = prefix_f64(tile_sums_f32(q))
    want = np.cumsum(np.pad(q, (0, (-len(q)) % TILE)).reshape(-1, TILE).sum(1))
    assert np.array_equal(got, want)


@pytest.mark.parametrize("V,scale", [(32000, 3.0), (128256, 3.0), (151936, 1.0)])
def test_drafting_prefix_error_bound(V, scale):
    """The kernel's prefix at every tile boundary is within 5e-7 W of the
    exact cumulative sum (float64 of the float32 row values) on draft rows
    of the workloads' kind (softmax of scaled Gaussian logits)."""
    rng = np.random.default_rng(V)
    worst = 0.0
    for _ in range(4):
        z = rng.standard_normal(V) * scale
        q = np.exp(z - z.max())
        q = (q / q.sum()).astype(np.float32).astype(np.float64)
        pre = prefix_f64(tile_sums_f32(q))
        exact = np.cumsum(np.pad(q, (0, (-V) % TILE)).reshape(-1, TILE).sum(1))
        W = exact[-1]
        worst = max(worst, float(np.max(np.abs(pre - exact)) / W))
    print(f"\nV={V}: worst prefix error {worst:.2e} W")
    assert worst < 5e-7
