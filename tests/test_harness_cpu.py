"""The oracle-side helpers of the GPU tests agree with each other on CPU:
the per-layer oracle that regenerates one sequence's pages at a time gives
exactly the rows of the oracle run over the whole regenerated pool."""
import numpy as np
import pytest

from wm_synth import configs
from wm_synth.inputs import make_problem

from . import _harness as H


@pytest.mark.parametrize("name,overrides,lens", [
    ("tiny_f32", dict(), None),
    ("no_compression", dict(B=3, L=2, k=2, permute_pages=True), [100, 17, 2048]),
    ("paper_k8", dict(B=2, L=3), [300, 2]),
])
def test_layer_oracle_equals_whole_pool_oracle(name, overrides, lens):
    w = configs.get(name).with_(**overrides)
    prob = make_problem(w, 0, lens)
    for layer in range(w.L):
        assert np.array_equal(H.oracle_attn_layer(prob, layer), H.oracle_attn_full(prob, layer))
