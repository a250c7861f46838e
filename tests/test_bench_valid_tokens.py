"""The valid-token share bench.py reports beside the transformer's dense
FLOP count: the mean sequence length over the resident batches, divided by
the padded length (lengths are drawn uniformly from 32..128, so the share
is near 80 / 128), and nothing for the image workloads."""
import numpy as np

import bench
from paper_2504_13850_gb300 import workloads as W


def test_valid_token_share_of_the_transformer_batches():
    cfg = W.CONFIGS["transformer"]
    f = bench.valid_token_frac(cfg)
    L = cfg["in_hwc"][0]
    lengths = np.concatenate([W.device_batch(cfg, j % cfg["K"], 10_000 + j)[3] for j in range(bench.POOL)])
    assert f == round(lengths.mean() / L, 4)
    # 256 draws from U{32..128}: standard deviation ~28 tokens, so the mean's
    # standard error is ~1.75 tokens (0.014 of 128); 0.06 is over four of them
    assert abs(f - 80 / 128) < 0.06
    assert bench.valid_token_frac(W.CONFIGS["vgg"]) is None
