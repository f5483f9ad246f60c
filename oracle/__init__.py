"""CPU oracle of the NITRO-D local-loss block training step (arXiv 2407.11698).

TEST INFRASTRUCTURE ONLY.  Plain, slow, obviously correct: the integer
contractions and element-wise pieces live in ``nitro_oracle.c`` (plain loops,
int64), this module strings them together in the order the paper trains a
block (Sec. 3.3 training iteration).  Only ``tests/``, the smoke check and the
benchmark's CPU-baseline leg may import it; the GPU library never does.

Every part is pinned to something other than itself by
``tests/test_oracle_pins.py`` and ``tests/test_oracle_lrpool_dropout.py``; no
part is parity unpinned.
"""
from .nitro import (  # noqa: F401
    FLOOR, TRUNC, ST_OVERFLOW, ST_BAD_LABEL, CONV, LINEAR,
    LayerDesc, OracleBlock, train_step, lib, fdiv, tdiv, relu_mu, relu, relu_region,
    relu_bwd, isqrt, init_bound, splitmix64_at, conv3x3_fwd, conv3x3_dgrad,
    conv3x3_wgrad, linear_fwd, linear_dgrad, linear_wgrad, maxpool_fwd, maxpool_bwd,
    integersgd, amplification_factor, num_threads, prep_stats, prep_apply,
    winpool_fwd, winpool_bwd, dropout_drop, dropout_mask, lr_pool_window, scale_relu,
)
