"""The seeded input generator: the torch-device variant used for the large
benchmark models reproduces the numpy generator the oracle uses."""
import numpy as np
import torch

import xc_inputs as X


def test_torch_generator_matches_numpy_counters_and_weights():
    for name, n, off in (("pin/a", 4000, 0), ("pin/b", 3000, 987654)):
        a = X.normal(5, name, n, offset=off)
        b = X.normal_torch(5, name, n, "cpu", offset=off, block=1024).numpy()
        # same counters and SplitMix64 bits; log / cos may differ in the last bit
        np.testing.assert_allclose(b, a, rtol=0, atol=4 * np.finfo(np.float64).eps * np.abs(a).max())
    for cfg in (X.MID_HD64, X.TINY_F32, X.XATTN_BF16):
        for k in X.weight_shapes(cfg):
            np.testing.assert_array_equal(X.make_weight_torch(cfg, k, "cpu").numpy(), X.make_weight(cfg, k))


def test_torch_generator_block_offsets():
    """Values do not depend on how the request is split into blocks."""
    a = X.normal_torch(1, "pin/c", 5000, "cpu", block=5000)
    b = X.normal_torch(1, "pin/c", 5000, "cpu", block=777)
    assert torch.equal(a, b)
