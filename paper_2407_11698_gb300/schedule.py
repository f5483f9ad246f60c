"""Inverse-learning-rate schedule of App. B: the learning rate is divided by 3,
i.e. gamma_inv multiplied by 3, each time the monitored test accuracy stops
improving.  Host-side bookkeeping only; the new value reaches the GPU through
``Block.set_hyper`` (``nitro_block_set_hyper``).

The appendix does not say when an accuracy counts as a plateau.  Reading used
here: after ``patience`` consecutive evaluations none of which beat the best
accuracy so far by more than ``min_delta``, gamma_inv is multiplied by
``factor`` (3) and the count starts again from zero.
"""


class GammaPlateau:
    def __init__(self, gamma_inv: int, factor: int = 3, patience: int = 5,
                 min_delta: float = 0.0, max_gamma_inv: int = 1 << 48):
        if gamma_inv < 1 or factor < 2 or patience < 1 or min_delta < 0:
            raise ValueError("gamma_inv >= 1, factor >= 2, patience >= 1, min_delta >= 0")
        self.gamma_inv = int(gamma_inv)
        self.factor = int(factor)
        self.patience = int(patience)
        self.min_delta = float(min_delta)
        self.max_gamma_inv = int(max_gamma_inv)
        self.best = None
        self.stale = 0
        self.reductions = 0

    def step(self, accuracy: float) -> bool:
        """Record one evaluation; returns True when gamma_inv was just raised."""
        if self.best is None or accuracy > self.best + self.min_delta:
            self.best = accuracy
            self.stale = 0
            return False
        self.stale += 1
        if self.stale < self.patience:
            return False
        self.stale = 0
        nxt = self.gamma_inv * self.factor
        if nxt > self.max_gamma_inv:
            return False
        self.gamma_inv = nxt
        self.reductions += 1
        return True

    def apply(self, blocks, eta_inv_fw: int = 0, eta_inv_lr: int = 0):
        """Push the current gamma_inv to every block handle."""
        for b in blocks:
            b.set_hyper(self.gamma_inv, eta_inv_fw, eta_inv_lr)
