"""GPU parity on large and deep trees: the Sequoia-scale deep768 workload
(768 nodes, depth 24), and batches whose trees all differ in shape, up to the
largest tree the library takes (N = 1023, 1024 rows)."""

import pytest
import torch

from tests.test_gpu_parity import check
from tests.test_gpu_tokenlevel import check as check_token
from workloads.synth import get_workload, make_inputs, make_inputs_random_shapes

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tv():
    import paper_2505_12398_gb300 as tv
    from paper_2505_12398_gb300.build import build
    build()
    return tv


@pytest.mark.parametrize("path", ["persistent", "three"])
def test_deep768(tv, path):
    w = get_workload("deep768", batch=16)
    inp = make_inputs(w, seed=31, device="cuda")
    check(tv, inp, trees=[0, 5, 10, 15], path=path)


@pytest.mark.parametrize("path", ["persistent", "three"])
def test_largest_trees_random_shapes(tv, path):
    """Eight trees of 1023 draft nodes, each of a different shape."""
    inp = make_inputs_random_shapes(8, 1023, 8192, seed=32, device="cuda")
    check(tv, inp, path=path)


def test_random_shapes_batch(tv):
    inp = make_inputs_random_shapes(96, 255, 32000, seed=33, device="cuda")
    check(tv, inp, trees=list(range(0, 96, 12)), path="persistent")


def test_random_shapes_token_level(tv):
    inp = make_inputs_random_shapes(96, 255, 32000, seed=34, device="cuda")
    check_token(tv, inp, "persistent", trees=list(range(0, 96, 12)))
