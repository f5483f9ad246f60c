"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

Holds none of the method's arithmetic: only the recipe for the integer images
and labels that stand in for MNIST / FashionMNIST / CIFAR-10 (Sec. 4 shapes:
28x28x1 and 32x32x3 images, G = 10 classes).  Images are int8 uniform on
[-128, 127]; labels uniform on [0, G).  Batch ``step`` of a run seeded with
``seed`` comes from numpy's PCG64 seeded by the pair (seed, step), so any step
can be regenerated on its own.
"""
import numpy as np


def _rng(seed: int, step: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, step, stream])))


def images(seed: int, step: int, batch: int, shape) -> np.ndarray:
    """int8 images of shape (batch, *shape), NHWC, uniform on [-128, 127]."""
    return _rng(seed, step, 0).integers(-128, 128, size=(batch, *shape), dtype=np.int8)


def labels(seed: int, step: int, batch: int, num_classes: int = 10) -> np.ndarray:
    """int32 class labels uniform on [0, num_classes)."""
    return _rng(seed, step, 1).integers(0, num_classes, size=(batch,), dtype=np.int32)


def gaussian_images(seed: int, step: int, batch: int, shape, sigma: float = 64.0) -> np.ndarray:
    """int8 images drawn as round(N(0, sigma^2)) clamped to [-128, 127]: the
    distribution App. A's preprocessing aims for (mean 0, sigma 64)."""
    x = np.rint(_rng(seed, step, 2).normal(0.0, sigma, size=(batch, *shape)))
    return np.clip(x, -128, 127).astype(np.int8)


def int_tensor(seed: int, shape, lo: int, hi: int, stream: int = 3, dtype=np.int64) -> np.ndarray:
    """Integer tensor uniform on [lo, hi] (inclusive), for kernel-level tests."""
    return _rng(seed, 0, stream).integers(lo, hi + 1, size=shape, dtype=dtype)


def raw_pixels(seed: int, n: int, kind: str = "natural") -> np.ndarray:
    """uint8 pixel values standing in for a raw 8-bit image dataset before
    pre-processing (App. A), flattened to n values:
      "natural"  round(N(120, 64^2)) clamped to [0, 255]: a broad, mid-grey
                 centred spread like CIFAR-10 photographs;
      "digits"   80% background zeros, the rest uniform on [1, 255]: mostly
                 empty strokes on black like MNIST / FashionMNIST;
      "uniform"  uniform on [0, 255];
      "constant" every value 77 (mean absolute deviation 0)."""
    r = _rng(seed, 0, 4)
    if kind == "natural":
        return np.clip(np.rint(r.normal(120.0, 64.0, size=n)), 0, 255).astype(np.uint8)
    if kind == "digits":
        x = r.integers(1, 256, size=n, dtype=np.int64)
        x[r.random(n) < 0.8] = 0
        return x.astype(np.uint8)
    if kind == "uniform":
        return r.integers(0, 256, size=n, dtype=np.uint8)
    if kind == "constant":
        return np.full(n, 77, dtype=np.uint8)
    raise ValueError(kind)
