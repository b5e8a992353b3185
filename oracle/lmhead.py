"""Logits of the target model's last layer and their row normalisers: the step
right before verification (the target distributions M_b(.|X^i) = softmax(l_i / T)
of §3.1 are computed from these logits) -- literal, float64, slow.

TEST INFRASTRUCTURE ONLY: imported by tests/, the smoke check and the CPU
legs of bench.py, never by the product path.

* logits l[r, v] = sum_k H[r, k] W[v, k]: the hidden state of row r times the
  output embedding of token v, in float64 from the given values;
* the stored logits are l rounded to bfloat16 (nearest, ties to even), the
  element type the verification reads;
* the normaliser of a stored row is (m, s) with m = max_v l[r, v] and
  s = sum_v 2^((l[r, v] - m) log2(e) / T), so that
  M_b(v) = 2^((l[r, v] - m) log2(e) / T) / s is the softmax of l / T.
"""

import numpy as np

LOG2E = 1.4426950408889634


def logits(hidden, weight):
    """l = H W^T in float64 ([rows, K] times [V, K] -> [rows, V])."""
    return np.asarray(hidden, dtype=np.float64) @ np.asarray(weight, dtype=np.float64).T


def to_bf16(x):
    """Rounds float64 values to the nearest bfloat16 (8 significant bits,
    ties to even), returned as float64; zeros stay zero."""
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)                 # x = f 2^e, 0.5 <= |f| < 1
    return np.ldexp(np.rint(f * 256.0) / 256.0, e)   # np.rint rounds half to even


def bf16_boundary_distance(x):
    """Distance from each value to the nearest point where rounding to
    bfloat16 changes direction (the midpoints between adjacent bfloat16
    values).  A computation whose error exceeds this distance may round
    either way."""
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)
    frac = np.abs(f) * 256.0           # in [128, 256): units of one bf16 step
    dist_steps = np.abs(frac - np.floor(frac) - 0.5)
    return dist_steps * np.ldexp(1.0, e - 8)


def row_stats(stored_logits, temperature):
    """(m, s) of every row of the stored logits, in float64."""
    l = np.asarray(stored_logits, dtype=np.float64)
    m = l.max(axis=-1)
    c = LOG2E / np.float64(temperature)
    s = np.exp2((l - m[..., None]) * c).sum(axis=-1)
    return m, s
