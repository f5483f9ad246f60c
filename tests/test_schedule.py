"""Host-side checks of the App. B inverse-learning-rate schedule (no GPU)."""
import pytest

from paper_2407_11698_gb300.schedule import GammaPlateau


def test_improving_accuracy_keeps_gamma():
    s = GammaPlateau(512, patience=2)
    for acc in (0.1, 0.2, 0.3, 0.4, 0.5):
        assert not s.step(acc)
    assert s.gamma_inv == 512 and s.reductions == 0


def test_plateau_multiplies_by_three_and_restarts_the_count():
    s = GammaPlateau(512, patience=3)
    seq = [0.50, 0.60, 0.60, 0.59, 0.60,   # 3 evaluations without a new best -> 1536
           0.58, 0.60, 0.55,               # 3 more -> 4608
           0.61, 0.61]                     # new best, then one stale
    raised = [s.step(a) for a in seq]
    assert raised == [False, False, False, False, True, False, False, True, False, False]
    assert s.gamma_inv == 512 * 9 and s.reductions == 2 and s.best == 0.61 and s.stale == 1


def test_min_delta_counts_small_gains_as_plateau():
    s = GammaPlateau(100, patience=2, min_delta=0.01)
    assert [s.step(a) for a in (0.5, 0.505, 0.509)] == [False, False, True]
    assert s.gamma_inv == 300


def test_ceiling_and_argument_checks():
    s = GammaPlateau(1 << 47, patience=1)
    s.step(0.5)
    assert not s.step(0.5)               # 3 * 2^47 would pass the 2^48 limit of the ABI
    assert s.gamma_inv == 1 << 47
    for kw in (dict(gamma_inv=0), dict(gamma_inv=5, factor=1), dict(gamma_inv=5, patience=0)):
        with pytest.raises(ValueError):
            GammaPlateau(**kw)


def test_apply_pushes_to_every_block():
    class Fake:
        def __init__(self):
            self.calls = []

        def set_hyper(self, g, efw, elr):
            self.calls.append((g, efw, elr))

    s = GammaPlateau(512, patience=1)
    blocks = [Fake(), Fake()]
    s.step(0.3)
    s.step(0.3)
    s.apply(blocks, eta_inv_fw=25000, eta_inv_lr=3000)
    assert [b.calls for b in blocks] == [[(1536, 25000, 3000)]] * 2
