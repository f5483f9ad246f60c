"""Block-level orchestration of the C oracle (test infrastructure only).

Every arithmetic step is a call into ``nitro_oracle.c``; this file fixes the
order of the steps, the shapes, and the points where a value is stored into its
declared integer type (the learning-pool window size and the selection of
dropped activations are plain Python on the C results).  Those storage rules are part of the definition the GPU
library must reproduce bit for bit:

* activations are int8 (NITRO-ReLU output, Sec. 3.2.2);
* gradients delta and the loss gradient are int32: a value that does not fit
  raises the OVERFLOW status and keeps its low 32 bits;
* weight gradients are int64 and weights int32 (same OVERFLOW rule on update);
* a contraction of two int32 tensors (delta_fw = grad_L W_lr, and dgrad) is
  exact in int64 only while max|A| * max|B| * K < 2^63; past that bound the
  OVERFLOW status is raised and the sum is kept modulo 2^64;
* the loss is floor(SSE / 2) with SSE summed modulo 2^64.
"""
import ctypes
from dataclasses import dataclass

import numpy as np

from . import build as _build

CONV, LINEAR = 0, 1
FLOOR, TRUNC = 0, 1
ST_OVERFLOW = 1
ST_BAD_LABEL = 2

LEARNING_TENSOR_ID = 255       # SplitMix64 stream of the learning / output layer
ONE_HOT_VALUE = 32             # scaled one-hot target (Sec. 3.3.4, App. A)

_I64 = ctypes.c_int64
_P64 = ctypes.POINTER(ctypes.c_int64)
_lib = None


def lib():
    """Load (building if needed) ``libnitro_oracle.so`` and declare its ABI."""
    global _lib
    if _lib is not None:
        return _lib
    L = ctypes.CDLL(_build.build())
    for name in ("nor_fdiv", "nor_tdiv"):
        getattr(L, name).argtypes = [_I64, _I64]
        getattr(L, name).restype = _I64
    L.nor_relu_mu.argtypes = [_I64]
    L.nor_relu_mu.restype = _I64
    L.nor_relu.argtypes = [_I64, _I64, _I64]
    L.nor_relu.restype = _I64
    L.nor_relu_region.argtypes = [_I64]
    L.nor_relu_region.restype = _I64
    L.nor_relu_bwd.argtypes = [_I64, _I64, _I64]
    L.nor_relu_bwd.restype = _I64
    L.nor_isqrt.argtypes = [_I64]
    L.nor_isqrt.restype = _I64
    L.nor_init_bound.argtypes = [_I64]
    L.nor_init_bound.restype = _I64
    L.nor_splitmix64_at.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
    L.nor_splitmix64_at.restype = ctypes.c_uint64
    L.nor_num_threads.argtypes = []
    L.nor_num_threads.restype = _I64
    L.nor_init_uniform.argtypes = [_I64, _I64, ctypes.c_uint64, ctypes.c_uint64, _P64]
    L.nor_fdiv_vec.argtypes = [_I64, _P64, _I64, _P64]
    L.nor_scale_relu.argtypes = [_I64, _P64, _I64, _I64, _P64, _P64, _P64]
    L.nor_relu_bwd_vec.argtypes = [_I64, _P64, _P64, _I64, _P64]
    for name in ("nor_conv3x3_fwd", "nor_conv3x3_dgrad", "nor_conv3x3_wgrad"):
        getattr(L, name).argtypes = [_I64] * 5 + [_P64, _P64, _P64]
    for name in ("nor_linear_fwd", "nor_linear_dgrad", "nor_linear_wgrad"):
        getattr(L, name).argtypes = [_I64] * 3 + [_P64, _P64, _P64]
    for name in ("nor_maxpool_fwd",):
        getattr(L, name).argtypes = [_I64] * 4 + [_P64, _P64, _P64]
    L.nor_maxpool_bwd.argtypes = [_I64] * 4 + [_P64, _P64, _P64]
    L.nor_winpool_fwd.argtypes = [_I64] * 6 + [_P64, _P64, _P64]
    L.nor_winpool_bwd.argtypes = [_I64] * 6 + [_P64, _P64, _P64]
    L.nor_dropout_drop.argtypes = [ctypes.c_uint64] * 4 + [_I64]
    L.nor_dropout_drop.restype = _I64
    L.nor_dropout_mask.argtypes = [_I64, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                   _I64, _P64]
    L.nor_integersgd.argtypes = [_I64, _P64, _P64, _I64, _I64, _I64]
    L.nor_prep_stats.argtypes = [_I64, ctypes.c_void_p, _P64, _P64]
    L.nor_prep_apply.argtypes = [_I64, ctypes.c_void_p, _I64, _I64, ctypes.c_void_p]
    _lib = L
    return L


def _c(a):
    """C-contiguous int64 copy-or-view of ``a``."""
    return np.ascontiguousarray(a, dtype=np.int64)


def _p(a):
    return a.ctypes.data_as(_P64)


# --------------------------------------------------------------------------
# scalar pieces (used by the pins)
# --------------------------------------------------------------------------
def fdiv(x, d):
    return lib().nor_fdiv(int(x), int(d))


def tdiv(x, d):
    return lib().nor_tdiv(int(x), int(d))


def relu_mu(alpha_inv):
    return lib().nor_relu_mu(int(alpha_inv))


def relu(x, alpha_inv):
    return lib().nor_relu(int(x), int(alpha_inv), relu_mu(alpha_inv))


def relu_region(x):
    return lib().nor_relu_region(int(x))


def relu_bwd(g, region, alpha_inv):
    return lib().nor_relu_bwd(int(g), int(region), int(alpha_inv))


def isqrt(n):
    return lib().nor_isqrt(int(n))


def init_bound(fan_in):
    return lib().nor_init_bound(int(fan_in))


def splitmix64_at(seed, index):
    return lib().nor_splitmix64_at(int(seed) & (2**64 - 1), int(index) & (2**64 - 1))


def num_threads():
    return lib().nor_num_threads()


def prep_stats(x):
    """(mu_int, omega_int) of the 8-bit values ``x`` (App. A)."""
    x = np.ascontiguousarray(x, dtype=np.uint8).reshape(-1)
    if x.size == 0:
        raise ValueError("pre-processing needs at least one value")
    mu, om = ctypes.c_int64(), ctypes.c_int64()
    lib().nor_prep_stats(x.size, x.ctypes.data, ctypes.byref(mu), ctypes.byref(om))
    return mu.value, om.value


def prep_apply(x, mu, omega):
    """x_hat = floor((x - mu) 51 / omega) as int8 in [-127, 127] (App. A)."""
    x = np.ascontiguousarray(x, dtype=np.uint8)
    out = np.empty(x.shape, dtype=np.int8)
    lib().nor_prep_apply(x.size, x.ctypes.data, int(mu), int(omega), out.ctypes.data)
    return out


def amplification_factor(num_classes):
    """NITRO Amplification Factor AF = 2^6 * G (Sec. 3.3.5)."""
    return 64 * int(num_classes)


# --------------------------------------------------------------------------
# vector pieces
# --------------------------------------------------------------------------
def fdiv_vec(x, d):
    x = _c(x)
    out = np.empty_like(x)
    lib().nor_fdiv_vec(x.size, _p(x), int(d), _p(out))
    return out


def scale_relu(z, sf, alpha_inv):
    """NITRO-Scaling then NITRO-ReLU; returns (z*, region code, activation)."""
    z = _c(z)
    zs, reg, act = np.empty_like(z), np.empty_like(z), np.empty_like(z)
    lib().nor_scale_relu(z.size, _p(z), int(sf), int(alpha_inv), _p(zs), _p(reg), _p(act))
    return zs, reg, act


def relu_bwd_vec(g, region, alpha_inv):
    g, region = _c(g), _c(region)
    out = np.empty_like(g)
    lib().nor_relu_bwd_vec(g.size, _p(g), _p(region), int(alpha_inv), _p(out))
    return out


def init_uniform(shape, bound, seed, tensor_id):
    n = int(np.prod(shape))
    w = np.empty(n, dtype=np.int64)
    lib().nor_init_uniform(n, int(bound), int(seed) & (2**64 - 1), int(tensor_id), _p(w))
    return w.reshape(shape)


def conv3x3_fwd(a, w):
    a, w = _c(a), _c(w)
    B, H, W, Cin = a.shape
    Cout = w.shape[0]
    assert w.shape == (Cout, 3, 3, Cin)
    z = np.empty((B, H, W, Cout), dtype=np.int64)
    lib().nor_conv3x3_fwd(B, H, W, Cin, Cout, _p(a), _p(w), _p(z))
    return z


def conv3x3_dgrad(g_out, w):
    g_out, w = _c(g_out), _c(w)
    B, H, W, Cout = g_out.shape
    Cin = w.shape[3]
    assert w.shape == (Cout, 3, 3, Cin)
    g_in = np.empty((B, H, W, Cin), dtype=np.int64)
    lib().nor_conv3x3_dgrad(B, H, W, Cin, Cout, _p(g_out), _p(w), _p(g_in))
    return g_in


def conv3x3_wgrad(a, g_out):
    a, g_out = _c(a), _c(g_out)
    B, H, W, Cin = a.shape
    Cout = g_out.shape[3]
    assert g_out.shape[:3] == (B, H, W)
    dw = np.empty((Cout, 3, 3, Cin), dtype=np.int64)
    lib().nor_conv3x3_wgrad(B, H, W, Cin, Cout, _p(a), _p(g_out), _p(dw))
    return dw


def linear_fwd(a, w):
    a, w = _c(a), _c(w)
    B, In = a.shape
    Out = w.shape[0]
    assert w.shape == (Out, In)
    z = np.empty((B, Out), dtype=np.int64)
    lib().nor_linear_fwd(B, In, Out, _p(a), _p(w), _p(z))
    return z


def linear_dgrad(g_out, w):
    g_out, w = _c(g_out), _c(w)
    B, Out = g_out.shape
    In = w.shape[1]
    assert w.shape == (Out, In)
    g_in = np.empty((B, In), dtype=np.int64)
    lib().nor_linear_dgrad(B, In, Out, _p(g_out), _p(w), _p(g_in))
    return g_in


def linear_wgrad(a, g_out):
    a, g_out = _c(a), _c(g_out)
    B, In = a.shape
    Out = g_out.shape[1]
    assert g_out.shape[0] == B
    dw = np.empty((Out, In), dtype=np.int64)
    lib().nor_linear_wgrad(B, In, Out, _p(a), _p(g_out), _p(dw))
    return dw


def maxpool_fwd(a):
    a = _c(a)
    B, H, W, C = a.shape
    out = np.empty((B, H // 2, W // 2, C), dtype=np.int64)
    am = np.empty_like(out)
    lib().nor_maxpool_fwd(B, H, W, C, _p(a), _p(out), _p(am))
    return out, am


def maxpool_bwd(g_out, argmax, H, W):
    g_out, argmax = _c(g_out), _c(argmax)
    B, _, _, C = g_out.shape
    g_in = np.empty((B, H, W, C), dtype=np.int64)
    lib().nor_maxpool_bwd(B, H, W, C, _p(g_out), _p(argmax), _p(g_in))
    return g_in


def winpool_fwd(a, kh, kw):
    """kh x kw max-pool, stride (kh, kw), first maximum in row-major window
    order; returns (pooled, argmax position r * kw + s)."""
    a = _c(a)
    B, H, W, C = a.shape
    out = np.empty((B, H // kh, W // kw, C), dtype=np.int64)
    am = np.empty_like(out)
    lib().nor_winpool_fwd(B, H, W, C, int(kh), int(kw), _p(a), _p(out), _p(am))
    return out, am


def winpool_bwd(g_out, argmax, H, W, kh, kw):
    g_out, argmax = _c(g_out), _c(argmax)
    B, _, _, C = g_out.shape
    g_in = np.empty((B, H, W, C), dtype=np.int64)
    lib().nor_winpool_bwd(B, H, W, C, int(kh), int(kw), _p(g_out), _p(argmax), _p(g_in))
    return g_in


def dropout_drop(seed, step, layer, e, p16):
    """1 if element e of forward layer ``layer`` is dropped at step ``step``."""
    return lib().nor_dropout_drop(int(seed) & (2**64 - 1), int(step), int(layer), int(e),
                                  int(p16))


def dropout_mask(n, seed, step, layer, p16):
    drop = np.empty(int(n), dtype=np.int64)
    lib().nor_dropout_mask(int(n), int(seed) & (2**64 - 1), int(step), int(layer), int(p16),
                           _p(drop))
    return drop


MAX_LR_WINDOW = 256     # positions of a learning-pool window (argmax kept in a byte)


def lr_pool_window(C, H, W, d_lr):
    """Window (kh, kw) of the learning-layer max-pool that brings a C x H x W
    block output down to at most d_lr features (App. B's d^lr; Sec. 3.3 names
    the pooled tensor z^mp).  Reading (the paper states no rule): starting
    from 1 x 1, double the window height, then its width, alternately, while
    C * floor(H / kh) * floor(W / kw) > d_lr and the window still fits the
    map; a side that can no longer double leaves the other to grow.  d_lr = 0
    means no pooling."""
    kh = kw = 1
    if d_lr <= 0:
        return 1, 1
    while C * (H // kh) * (W // kw) > d_lr:
        if kh <= kw and 2 * kh <= H:
            kh *= 2
        elif 2 * kw <= W:
            kw *= 2
        elif 2 * kh <= H:
            kh *= 2
        else:
            break
    return kh, kw


def integersgd(w, dw, gamma_inv, eta_inv, round_mode=FLOOR):
    """Algorithm 1 on a copy of ``w``; returns the int64 result (unchecked)."""
    w = _c(w).copy()
    dw = _c(dw)
    assert w.shape == dw.shape
    lib().nor_integersgd(w.size, _p(w), _p(dw), int(gamma_inv), int(eta_inv), int(round_mode))
    return w


# --------------------------------------------------------------------------
# storage rules
# --------------------------------------------------------------------------
def store32(x):
    """Store into int32: (low-32-bit value, True if the value did not fit)."""
    x = _c(x)
    bad = bool(np.any((x < -2**31) | (x > 2**31 - 1))) if x.size else False
    return x.astype(np.int32).astype(np.int64), bad


def maxabs(x):
    return int(np.abs(_c(x)).max()) if np.size(x) else 0


def int64_bound_exceeded(a, b, k):
    """True when max|a| * max|b| * k >= 2^63 (int64 exactness not guaranteed)."""
    return maxabs(a) * maxabs(b) * int(k) >= 2**63


# --------------------------------------------------------------------------
# block description
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class LayerDesc:
    """One forward layer: 3x3 conv (stride 1, pad 1) or linear, then
    NITRO-Scaling and NITRO-ReLU, then an optional 2x2 max-pool (conv only).
    ``h``/``w`` are the layer's input spatial size (1 for linear)."""
    kind: int
    cin: int
    cout: int
    h: int = 1
    w: int = 1
    pool: bool = False

    @property
    def out_hw(self):
        if self.kind == LINEAR:
            return 1, 1
        return (self.h // 2, self.w // 2) if self.pool else (self.h, self.w)

    @property
    def in_features(self):
        return self.h * self.w * self.cin

    @property
    def out_features(self):
        oh, ow = self.out_hw
        return oh * ow * self.cout

    @property
    def fan_in(self):
        return 9 * self.cin if self.kind == CONV else self.cin

    @property
    def scaling_factor(self):
        """SF = 2^8 * K^2 * C_in (conv) or 2^8 * M (linear), Sec. 3.2.1."""
        return 256 * self.fan_in

    @property
    def w_shape(self):
        return (self.cout, 3, 3, self.cin) if self.kind == CONV else (self.cout, self.cin)


class OracleBlock:
    """One integer local-loss block (Sec. 3.2): forward layers, then a learning
    layer (max-pool to at most d_lr features, or identity -> IntLinear(d -> G)
    -> NITRO-Scaling) trained on the RSS loss against the scaled one-hot
    target.  A block with no forward layers is the network's output block: its
    learning layer is the output layer.  dropout_p16 > 0 drops the outputs of
    the block's linear forward layers during training (App. B's p_l, in units
    of 2^-16); the mask of step t comes from the block's SplitMix64 stream,
    and t counts the IntegerSGD steps the block has taken."""

    def __init__(self, layers, in_features=None, num_classes=10, alpha_inv=10,
                 gamma_inv_lr=512, eta_inv_fw=0, eta_inv_lr=0, sgd_round=FLOOR,
                 seed=0, lr_post_update=False, d_lr=0, dropout_p16=0):
        self.layers = list(layers)
        self.seed = int(seed)
        self.dropout_p16 = int(dropout_p16)
        if not 0 <= self.dropout_p16 <= 65536:
            raise ValueError("dropout_p16 must lie in [0, 65536]")
        self.t = 0
        self.G = int(num_classes)
        self.alpha_inv = int(alpha_inv)
        self.gamma_inv_lr = int(gamma_inv_lr)
        self.eta_inv_fw = int(eta_inv_fw)
        self.eta_inv_lr = int(eta_inv_lr)
        self.sgd_round = int(sgd_round)
        # Reading kept only as an oracle option: delta_fw from the already
        # updated learning weights (the default uses the pre-update ones).
        self.lr_post_update = bool(lr_post_update)
        if self.alpha_inv < 2:
            raise ValueError("alpha_inv must be >= 2 for int8 activations")
        prev = None
        for L in self.layers:
            if L.kind == LINEAR and (L.h != 1 or L.w != 1 or L.pool):
                raise ValueError("linear layers take h = w = 1 and no pool")
            if prev is not None and L.in_features != prev.out_features:
                raise ValueError("layer input size does not match previous output")
            prev = L
        # learning-layer pooling window over the block output (conv blocks)
        self.lr_win = (1, 1)
        if self.layers:
            self.in_features = self.layers[0].in_features
            last = self.layers[-1]
            oh, ow = last.out_hw
            self.lr_win = lr_pool_window(last.cout, oh, ow, int(d_lr))
            kh, kw = self.lr_win
            if kh * kw > MAX_LR_WINDOW:
                raise ValueError("learning-pool window above %d positions" % MAX_LR_WINDOW)
            self.d = last.cout * (oh // kh) * (ow // kw)
        else:
            if not in_features:
                raise ValueError("an output block needs in_features")
            self.in_features = int(in_features)
            self.d = self.in_features
        # Integer Kaiming initialisation (Sec. 3.3.1), one SplitMix64 stream
        # per tensor.
        self.W = [init_uniform(L.w_shape, init_bound(L.fan_in), seed, i)
                  for i, L in enumerate(self.layers)]
        self.Wlr = init_uniform((self.G, self.d), init_bound(self.d), seed,
                                LEARNING_TENSOR_ID)
        self.dW = [np.zeros(L.w_shape, dtype=np.int64) for L in self.layers]
        self.dWlr = np.zeros((self.G, self.d), dtype=np.int64)
        self.status = 0

    # ------------------------------------------------------------------
    @property
    def gamma_inv_fw(self):
        """gamma_inv^fw = AF * gamma_inv^lr (Sec. 3.3.5)."""
        return amplification_factor(self.G) * self.gamma_inv_lr

    def forward(self, a_in):
        """Forward layers only (Sec. 3.3 training iteration, first phase).
        Returns the block output, flattened per sample, as int64 values."""
        a_in = _c(a_in)
        B = a_in.shape[0]
        if a_in.size != B * self.in_features:
            raise ValueError("input size mismatch")
        x = a_in.reshape(B, self.in_features)
        self.layer_in, self.zs, self.region, self.argmax, self.act = [], [], [], [], []
        for i, L in enumerate(self.layers):
            self.layer_in.append(x)
            if L.kind == CONV:
                z = conv3x3_fwd(x.reshape(B, L.h, L.w, L.cin), self.W[i])
            else:
                z = linear_fwd(x.reshape(B, L.cin), self.W[i])
            zs, reg, act = scale_relu(z, L.scaling_factor, self.alpha_inv)
            if L.kind == LINEAR and self.dropout_p16:
                # dropped outputs become 0 and carry region code 4, whose
                # NITRO-ReLU backward passes nothing
                drop = dropout_mask(act.size, self.seed, self.t, i,
                                    self.dropout_p16).reshape(act.shape)
                act = np.where(drop == 1, 0, act)
                reg = np.where(drop == 1, 4, reg)
            self.zs.append(zs)
            self.region.append(reg)
            if L.pool:
                act, am = maxpool_fwd(act)
                self.argmax.append(am)
            else:
                self.argmax.append(None)
            x = act.reshape(B, L.out_features)
            self.act.append(x)
        self.out = x
        self.batch = B
        return x

    def backward(self, a_in, labels):
        """Learning-layer forward, loss, and every weight gradient of the block
        (Sec. 3.3 second phase).  Returns floor(SSE / 2)."""
        labels = np.asarray(labels, dtype=np.int64).reshape(-1)
        self.lr_in, self.lr_argmax = None, None
        if self.layers:
            a = self.out
            if self.lr_win != (1, 1):
                # z^mp: the block output max-pooled for the learning layer
                last = self.layers[-1]
                oh, ow = last.out_hw
                zmp, am = winpool_fwd(a.reshape(a.shape[0], oh, ow, last.cout), *self.lr_win)
                a = zmp.reshape(a.shape[0], self.d)
                self.lr_in, self.lr_argmax = a, am.reshape(a.shape[0], self.d)
        else:
            a = _c(a_in).reshape(labels.size, self.in_features)
            self.batch = a.shape[0]
        B = a.shape[0]
        if labels.size != B:
            raise ValueError("labels / batch mismatch")
        # learning layer: IntLinear(d -> G) then NITRO-Scaling by 2^8 * d
        z = linear_fwd(a, self.Wlr)
        self.yhat = fdiv_vec(z, 256 * self.d)
        y = np.zeros((B, self.G), dtype=np.int64)
        for b in range(B):
            if 0 <= labels[b] < self.G:
                y[b, labels[b]] = ONE_HOT_VALUE
            else:
                self.status |= ST_BAD_LABEL
        # RSS loss and its per-sample gradient grad_L = yhat - y (Sec. 3.3.2)
        gl, bad = store32(self.yhat - y)
        self.status |= ST_OVERFLOW if bad else 0
        self.grad_l = gl
        sse = sum(int(v) * int(v) for v in gl.reshape(-1)) % 2**64
        self.sse = sse - 2**64 if sse >= 2**63 else sse
        self.loss = fdiv(self.sse, 2)
        # learning-layer weight gradient, from the block's own activations
        self.dWlr = linear_wgrad(a, gl)
        self.delta = [None] * len(self.layers)
        if not self.layers:
            return self.loss
        # delta_fw = grad_L W_lr (Sec. 3.3.5), pre-update learning weights
        wlr = self.Wlr
        if self.lr_post_update:
            wlr = self._updated(self.Wlr, self.dWlr, self.gamma_inv_lr, self.eta_inv_lr)
        if int64_bound_exceeded(gl, wlr, self.G):
            self.status |= ST_OVERFLOW
        g, bad = store32(linear_dgrad(gl, wlr))
        self.status |= ST_OVERFLOW if bad else 0
        if self.lr_in is not None:
            # back through the learning-layer pooling to the block output
            last = self.layers[-1]
            oh, ow = last.out_hw
            kh, kw = self.lr_win
            g = winpool_bwd(g.reshape(B, oh // kh, ow // kw, last.cout),
                            self.lr_argmax.reshape(B, oh // kh, ow // kw, last.cout),
                            oh, ow, kh, kw).reshape(B, last.out_features)
        # down through the forward layers: pool backward, ReLU backward, STE
        # through NITRO-Scaling (Sec. 3.2.1), weight gradient, input gradient
        for i in reversed(range(len(self.layers))):
            L = self.layers[i]
            if L.kind == CONV:
                oh, ow = L.out_hw
                g = g.reshape(B, oh, ow, L.cout)
                if L.pool:
                    g = maxpool_bwd(g, self.argmax[i], L.h, L.w)
            delta = relu_bwd_vec(g, self.region[i], self.alpha_inv)
            self.delta[i] = delta
            if L.kind == CONV:
                self.dW[i] = conv3x3_wgrad(self.layer_in[i].reshape(B, L.h, L.w, L.cin), delta)
            else:
                self.dW[i] = linear_wgrad(self.layer_in[i], delta)
            if i > 0:
                k = 9 * L.cout if L.kind == CONV else L.cout
                if int64_bound_exceeded(delta, self.W[i], k):
                    self.status |= ST_OVERFLOW
                if L.kind == CONV:
                    g = conv3x3_dgrad(delta, self.W[i])
                else:
                    g = linear_dgrad(delta, self.W[i])
                g, bad = store32(g.reshape(B, L.in_features))
                self.status |= ST_OVERFLOW if bad else 0
        return self.loss

    def _updated(self, w, dw, gamma_inv, eta_inv):
        return integersgd(w, dw, gamma_inv, eta_inv, self.sgd_round)

    def sgd(self):
        """IntegerSGD (Algorithm 1): forward layers with gamma_inv^fw = AF *
        gamma_inv^lr and eta_inv^fw; the learning layer with gamma_inv^lr and
        eta_inv^lr."""
        for i in range(len(self.layers)):
            w, bad = store32(self._updated(self.W[i], self.dW[i], self.gamma_inv_fw,
                                           self.eta_inv_fw))
            self.W[i] = w.reshape(self.layers[i].w_shape)
            self.status |= ST_OVERFLOW if bad else 0
        w, bad = store32(self._updated(self.Wlr, self.dWlr, self.gamma_inv_lr,
                                       self.eta_inv_lr))
        self.Wlr = w.reshape(self.G, self.d)
        self.status |= ST_OVERFLOW if bad else 0
        self.t += 1


def train_step(blocks, x, labels):
    """One training iteration (Sec. 3.3): forward through every block, then
    each block's local backward (independent: no gradient crosses blocks),
    then every update.  Returns the per-block losses."""
    acts = [_c(x)]
    for blk in blocks:
        acts.append(blk.forward(acts[-1]))
    losses = [blk.backward(acts[i], labels) for i, blk in enumerate(blocks)]
    for blk in blocks:
        blk.sgd()
    return losses
