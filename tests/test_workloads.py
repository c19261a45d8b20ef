"""Host checks of the seeded stack generators (no GPU): the packed weight layout they hand the
library is the oracle's (reading R6), and their draws are reproducible."""

import numpy as np

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import workloads as W


def test_packed_layout_matches_oracle():
    codes = W.gaussian_codes(np.random.default_rng(0), 8, 64)
    assert codes.min() >= -7 and codes.max() <= 7
    assert np.array_equal(W.pack_nibbles(codes), O.pack_int4(codes))
    packed = np.random.default_rng(1).integers(0, 256, (8, 32), dtype=np.uint8)
    sw = W.StackWeights("x", 64, 8, 64, packed, np.ones(8, np.float32), None)
    assert np.array_equal(sw.weight_codes(), O.unpack_int4(packed))


def test_stack_inputs_reproducible_and_independent():
    a = W.dit_layer_input(2, 5, 3, 4, 64)
    assert np.array_equal(a, W.dit_layer_input(2, 5, 3, 4, 64))
    assert not np.array_equal(a, W.dit_layer_input(2, 5, 4, 4, 64))
    # the step magnitude drifts from 4.0 to 0.5
    big = W.dit_layer_input(2, 0, 0, 256, 1024)
    small = W.dit_layer_input(2, 0, 9, 256, 1024)
    assert 3.8 < big.std() < 4.2 and 0.47 < small.std() < 0.53
    b = W.backbone_layer_input(3, 1, 8, 2048)
    assert np.array_equal(b, W.backbone_layer_input(3, 1, 8, 2048))
    assert np.count_nonzero(np.abs(b).max(0) > 15) >= 1


def test_stack_shapes():
    names = [(w.name, w.k, w.n, w.gated) for w in W.backbone_stack(layers=1)]
    assert names == [("0.qkv", 2048, 2560, False), ("0.o", 2048, 2048, False), ("0.gate_up", 2048, 16384, True),
                     ("0.down", 16384, 2048, False)]
