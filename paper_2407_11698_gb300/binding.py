"""ctypes binding of ``libnitro.so`` (declared in ``include/nitro.h``).

Argument marshalling only: every step of the block training step runs in the
library's CUDA kernels.  The module-level functions carry the C-ABI names and
return its status codes; ``Block`` wraps one handle for callers that hold
their activations and labels in torch CUDA tensors.  There is no CPU path:
loading fails loudly when the library has not been built.
"""
import ctypes
import os

import numpy as np

from . import build as _build

NITRO_OK, NITRO_ERR_ARG, NITRO_ERR_OVERFLOW, NITRO_ERR_TIMEOUT, NITRO_ERR_CUDA, \
    NITRO_ERR_UNSUPPORTED = range(6)
NITRO_CONV3X3, NITRO_LINEAR = 0, 1
NITRO_ROUND_FLOOR, NITRO_ROUND_TRUNC = 0, 1
STATUS_BIT_OVERFLOW, STATUS_BIT_BAD_LABEL, STATUS_BIT_TIMEOUT = 1, 2, 4
NITRO_CONTRACT_FWD, NITRO_CONTRACT_WGRAD, NITRO_CONTRACT_DGRAD = 0, 1, 2
(NITRO_T_W, NITRO_T_DW, NITRO_T_WLR, NITRO_T_DWLR, NITRO_T_ACT, NITRO_T_REGION,
 NITRO_T_ARGMAX, NITRO_T_DELTA, NITRO_T_GRAD_L, NITRO_T_SSE, NITRO_T_LR_IN, NITRO_T_LR_ARGMAX,
 NITRO_T_STEP) = range(13)

TENSOR_DTYPE = {
    NITRO_T_W: np.int32, NITRO_T_DW: np.int64, NITRO_T_WLR: np.int32, NITRO_T_DWLR: np.int64,
    NITRO_T_ACT: np.int8, NITRO_T_REGION: np.int8, NITRO_T_ARGMAX: np.int8,
    NITRO_T_DELTA: np.int32, NITRO_T_GRAD_L: np.int32, NITRO_T_SSE: np.int64,
    NITRO_T_LR_IN: np.int8, NITRO_T_LR_ARGMAX: np.uint8, NITRO_T_STEP: np.uint32,
}


class nitro_layer_desc(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("cin", ctypes.c_int), ("cout", ctypes.c_int),
                ("h", ctypes.c_int), ("w", ctypes.c_int), ("pool2x2", ctypes.c_int)]


class nitro_block_desc(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("layers", ctypes.POINTER(nitro_layer_desc)),
                ("in_features", ctypes.c_int), ("num_classes", ctypes.c_int),
                ("alpha_inv", ctypes.c_int), ("gamma_inv_lr", ctypes.c_int64),
                ("eta_inv_fw", ctypes.c_int64), ("eta_inv_lr", ctypes.c_int64),
                ("sgd_round", ctypes.c_int), ("max_batch", ctypes.c_int),
                ("d_lr", ctypes.c_int), ("dropout_p16", ctypes.c_int)]


class NitroError(RuntimeError):
    def __init__(self, status, what=""):
        self.status = int(status)
        super().__init__("%s: %s (status %d)" % (what, status_str(status), int(status)))


_lib = None
_VP = ctypes.c_void_p


def lib():
    """The loaded ``libnitro.so``; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB):
        raise RuntimeError("libnitro.so is missing (%s): build it with "
                           "paper_2407_11698_gb300.build.build() first" % _build.LIB)
    L = ctypes.CDLL(_build.LIB)
    L.nitro_init_block.argtypes = [ctypes.POINTER(nitro_block_desc), ctypes.c_uint64, _VP,
                                   ctypes.POINTER(_VP)]
    L.nitro_block_forward.argtypes = [_VP, _VP, ctypes.c_int, _VP, _VP]
    L.nitro_block_backward.argtypes = [_VP, _VP, _VP, ctypes.c_int, _VP, _VP]
    L.nitro_integersgd_step.argtypes = [_VP, _VP]
    L.nitro_block_backward_update.argtypes = [_VP, _VP, _VP, ctypes.c_int, _VP, _VP]
    L.nitro_block_tensor_bytes.argtypes = [_VP, ctypes.c_int, ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_size_t)]
    L.nitro_block_get_tensor.argtypes = [_VP, ctypes.c_int, ctypes.c_int, _VP, ctypes.c_size_t]
    L.nitro_block_set_tensor.argtypes = [_VP, ctypes.c_int, ctypes.c_int, _VP, ctypes.c_size_t]
    L.nitro_block_status.argtypes = [_VP, ctypes.c_int]
    L.nitro_block_status_bits.argtypes = [_VP]
    L.nitro_block_status_bits.restype = ctypes.c_uint32
    L.nitro_destroy_block.argtypes = [_VP]
    L.nitro_destroy_block.restype = None
    L.nitro_status_str.argtypes = [ctypes.c_int]
    L.nitro_status_str.restype = ctypes.c_char_p
    L.nitro_kernel_launches.argtypes = []
    L.nitro_kernel_launches.restype = ctypes.c_uint64
    L.nitro_profile_enable.argtypes = [ctypes.c_int]
    L.nitro_profile_enable.restype = None
    L.nitro_profile_reset.argtypes = []
    L.nitro_profile_reset.restype = None
    L.nitro_profile_kernel_count.argtypes = []
    L.nitro_profile_kernel_count.restype = ctypes.c_int
    L.nitro_profile_kernel_name.argtypes = [ctypes.c_int]
    L.nitro_profile_kernel_name.restype = ctypes.c_char_p
    _PD = ctypes.POINTER(ctypes.c_double)
    L.nitro_profile_read.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_uint64), _PD, _PD, _PD]
    L.nitro_profile_read.restype = ctypes.c_int
    L.nitro_profile_record_count.argtypes = []
    L.nitro_profile_record_count.restype = ctypes.c_int
    L.nitro_profile_record.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_int), _PD, _PD, _PD]
    L.nitro_profile_record.restype = ctypes.c_int
    L.nitro_conv3x3_forward_noalloc.argtypes = [_VP, _VP] + [ctypes.c_int] * 7 + [_VP, _VP, _VP, _VP]
    L.nitro_conv3x3_forward_noalloc.restype = ctypes.c_int
    L.nitro_conv3x3_create.argtypes = [ctypes.c_int] * 5 + [ctypes.POINTER(_VP)]
    L.nitro_conv3x3_contract.argtypes = [_VP, ctypes.c_int, _VP, _VP, ctypes.c_int, _VP, _VP]
    L.nitro_conv3x3_status.argtypes = [_VP]
    L.nitro_conv3x3_destroy.argtypes = [_VP]
    L.nitro_conv3x3_destroy.restype = None
    L.nitro_gemm_create.argtypes = [ctypes.c_int] * 3 + [ctypes.POINTER(_VP)]
    L.nitro_gemm_run.argtypes = [_VP, _VP, _VP, ctypes.c_int, ctypes.c_int, ctypes.c_int, _VP, _VP]
    L.nitro_gemm_status.argtypes = [_VP]
    L.nitro_gemm_destroy.argtypes = [_VP]
    L.nitro_gemm_destroy.restype = None
    L.nitro_block_set_hyper.argtypes = [_VP, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64]
    L.nitro_block_set_hyper.restype = ctypes.c_int
    L.nitro_block_set_dropout.argtypes = [_VP, ctypes.c_int]
    L.nitro_block_set_dropout.restype = ctypes.c_int
    L.nitro_block_diag_timeout.argtypes = [_VP, ctypes.c_int, _VP]
    L.nitro_block_diag_timeout.restype = ctypes.c_int
    L.nitro_block_grad_device.argtypes = [_VP, ctypes.c_int, ctypes.c_int, ctypes.POINTER(_VP),
                                          ctypes.POINTER(ctypes.c_size_t)]
    L.nitro_block_grad_device.restype = ctypes.c_int
    L.nitro_prep_create.argtypes = [ctypes.POINTER(_VP)]
    L.nitro_prep_fit.argtypes = [_VP, _VP, ctypes.c_int64, _VP]
    L.nitro_prep_apply.argtypes = [_VP, _VP, ctypes.c_int64, _VP, _VP]
    L.nitro_prep_stats.argtypes = [_VP, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
    L.nitro_prep_destroy.argtypes = [_VP]
    L.nitro_prep_destroy.restype = None
    for name in ("nitro_conv3x3_create", "nitro_conv3x3_contract", "nitro_conv3x3_status",
                 "nitro_gemm_create", "nitro_gemm_run", "nitro_gemm_status",
                 "nitro_prep_create", "nitro_prep_fit", "nitro_prep_apply", "nitro_prep_stats"):
        getattr(L, name).restype = ctypes.c_int
    for name in ("nitro_init_block", "nitro_block_forward", "nitro_block_backward",
                 "nitro_block_backward_update", "nitro_integersgd_step", "nitro_block_tensor_bytes", "nitro_block_get_tensor",
                 "nitro_block_set_tensor", "nitro_block_status"):
        getattr(L, name).restype = ctypes.c_int
    _lib = L
    return L


def status_str(s):
    try:
        return lib().nitro_status_str(int(s)).decode()
    except RuntimeError:
        return "status"


# ---------------------------------------------------------------- C-ABI names
def nitro_init_block(desc, seed, stream=None):
    """Returns (status, handle)."""
    h = _VP()
    st = lib().nitro_init_block(ctypes.byref(desc), int(seed) & (2**64 - 1), stream, ctypes.byref(h))
    return st, h


def nitro_block_forward(blk, a_in, batch, a_out, stream=None):
    return lib().nitro_block_forward(blk, a_in, int(batch), a_out, stream)


def nitro_block_backward(blk, a_in, labels, batch, loss_dev, stream=None):
    return lib().nitro_block_backward(blk, a_in, labels, int(batch), loss_dev, stream)


def nitro_integersgd_step(blk, stream=None):
    return lib().nitro_integersgd_step(blk, stream)


def nitro_block_backward_update(blk, a_in, labels, batch, loss_dev, stream=None):
    return lib().nitro_block_backward_update(blk, a_in, labels, int(batch), loss_dev, stream)


def nitro_block_tensor_bytes(blk, which, layer=0):
    n = ctypes.c_size_t()
    st = lib().nitro_block_tensor_bytes(blk, int(which), int(layer), ctypes.byref(n))
    return st, n.value


def nitro_block_get_tensor(blk, which, layer, host_ptr, nbytes):
    return lib().nitro_block_get_tensor(blk, int(which), int(layer), host_ptr, int(nbytes))


def nitro_block_set_tensor(blk, which, layer, host_ptr, nbytes):
    return lib().nitro_block_set_tensor(blk, int(which), int(layer), host_ptr, int(nbytes))


def nitro_block_status(blk, clear=False):
    return lib().nitro_block_status(blk, 1 if clear else 0)


def nitro_block_status_bits(blk):
    return lib().nitro_block_status_bits(blk)


def nitro_conv3x3_forward_noalloc(a_in, weights, batch, h, w, cin, cout, pool2x2, alpha_inv,
                                  a_out, region, argmax, stream=None):
    return lib().nitro_conv3x3_forward_noalloc(a_in, weights, int(batch), int(h), int(w), int(cin),
                                               int(cout), int(pool2x2), int(alpha_inv), a_out,
                                               region, argmax, stream)


def nitro_destroy_block(blk):
    lib().nitro_destroy_block(blk)


# ---------------------------------------------------------------- helpers
def make_block_desc(layers, in_features, num_classes=10, alpha_inv=10, gamma_inv_lr=512,
                    eta_inv_fw=0, eta_inv_lr=0, sgd_round=NITRO_ROUND_FLOOR, max_batch=1,
                    d_lr=0, dropout_p16=0):
    """Build a ``nitro_block_desc`` from layer tuples (kind, cin, cout, h, w, pool).
    Returns (desc, keepalive) - keep the second value alive while desc is used."""
    arr = (nitro_layer_desc * max(1, len(layers)))()
    for i, l in enumerate(layers):
        arr[i] = nitro_layer_desc(*[int(v) for v in l])
    d = nitro_block_desc(len(layers), arr if layers else None, int(in_features), int(num_classes),
                         int(alpha_inv), int(gamma_inv_lr), int(eta_inv_fw), int(eta_inv_lr),
                         int(sgd_round), int(max_batch), int(d_lr), int(dropout_p16))
    return d, arr


class _DeviceArray:
    """A 1-D device buffer described by __cuda_array_interface__ (so torch can
    view library-owned memory without copying it)."""

    def __init__(self, ptr, n, typestr):
        self.__cuda_array_interface__ = {"shape": (int(n),), "typestr": typestr,
                                         "data": (int(ptr or 0), False), "version": 3,
                                         "strides": None}


def _stream_ptr(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return _VP(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _ptr(t):
    return None if t is None else _VP(t.data_ptr())


class Block:
    """One local-loss block handle.  Activations / labels / loss are torch CUDA
    tensors (int8 / int32 / int64); calls queue work on the given (or current)
    torch stream."""

    def __init__(self, layers, in_features, seed=0, max_batch=1, stream=None, **hyper):
        self.layers = [tuple(int(v) for v in l) for l in layers]
        self.desc, self._keep = make_block_desc(self.layers, in_features, max_batch=max_batch,
                                                **hyper)
        st, self.h = nitro_init_block(self.desc, seed, _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_init_block")
        self.in_features = int(in_features)
        self.num_classes = self.desc.num_classes
        if self.layers:
            k, cin, cout, h, w, pool = self.layers[-1]
            self.out_features = (h // 2) * (w // 2) * cout if pool else h * w * cout
        else:
            self.out_features = 0

    def forward(self, a_in, a_out=None, stream=None):
        st = nitro_block_forward(self.h, _ptr(a_in), a_in.shape[0], _ptr(a_out), _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_forward")
        return a_out

    def backward(self, a_in, labels, loss=None, stream=None):
        st = nitro_block_backward(self.h, _ptr(a_in), _ptr(labels), labels.shape[0], _ptr(loss),
                                  _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_backward")
        return loss

    def backward_update(self, a_in, labels, loss=None, stream=None):
        """backward() then sgd() in one call, the update fused into the
        tensor-core weight-gradient kernels (same results)."""
        st = nitro_block_backward_update(self.h, _ptr(a_in), _ptr(labels), labels.shape[0],
                                         _ptr(loss), _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_backward_update")
        return loss

    def sgd(self, stream=None):
        st = nitro_integersgd_step(self.h, _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_integersgd_step")

    def set_hyper(self, gamma_inv_lr, eta_inv_fw=0, eta_inv_lr=0):
        st = lib().nitro_block_set_hyper(self.h, int(gamma_inv_lr), int(eta_inv_fw),
                                         int(eta_inv_lr))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_set_hyper")

    def set_dropout(self, dropout_p16):
        st = lib().nitro_block_set_dropout(self.h, int(dropout_p16))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_set_dropout")

    def get(self, which, layer=0, check=True):
        """Host copy of a tensor as a flat numpy array (synchronises)."""
        st, n = nitro_block_tensor_bytes(self.h, which, layer)
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_tensor_bytes")
        dt = np.dtype(TENSOR_DTYPE[which])
        out = np.empty(n // dt.itemsize, dtype=dt)
        st = nitro_block_get_tensor(self.h, which, layer, out.ctypes.data_as(_VP), n)
        if check and st not in (NITRO_OK,):
            raise NitroError(st, "nitro_block_get_tensor")
        return out

    def set(self, which, layer, values):
        dt = np.dtype(TENSOR_DTYPE[which])
        arr = np.ascontiguousarray(values, dtype=dt)
        st = nitro_block_set_tensor(self.h, which, layer, arr.ctypes.data_as(_VP), arr.nbytes)
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_set_tensor")

    def status(self, clear=False):
        return nitro_block_status(self.h, clear)

    def grad_device(self, which, layer=0):
        """The block's int64 weight gradient (NITRO_T_DW / NITRO_T_DWLR) as a
        flat torch CUDA tensor that views the block's own memory (no copy)."""
        import torch
        p, n = _VP(), ctypes.c_size_t()
        st = lib().nitro_block_grad_device(self.h, int(which), int(layer), ctypes.byref(p),
                                           ctypes.byref(n))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_grad_device")
        return torch.as_tensor(_DeviceArray(p.value, n.value // 8, "<i8"), device="cuda")

    def diag_timeout(self, wait_us, stream=None):
        """Queue the bounded-wait failure check (nitro_block_diag_timeout)."""
        st = lib().nitro_block_diag_timeout(self.h, int(wait_us), _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_block_diag_timeout")

    def status_bits(self):
        return nitro_block_status_bits(self.h)

    def close(self):
        if getattr(self, "h", None):
            nitro_destroy_block(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Conv3x3:
    """One 3x3 conv layer's contractions (kernel-level entry points)."""

    def __init__(self, max_batch, h, w, cin, cout):
        self.h = _VP()
        st = lib().nitro_conv3x3_create(int(max_batch), int(h), int(w), int(cin), int(cout),
                                        ctypes.byref(self.h))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_conv3x3_create")

    def contract(self, mode, x, y, out, stream=None):
        st = lib().nitro_conv3x3_contract(self.h, int(mode), _ptr(x), _ptr(y), int(x.shape[0]),
                                          _ptr(out), _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_conv3x3_contract")
        return out

    def status(self):
        return lib().nitro_conv3x3_status(self.h)

    def close(self):
        if getattr(self, "h", None):
            lib().nitro_conv3x3_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class IntGemm:
    """C = A B^T with A int8 [M][K], B int32 [N][K], C int64 (kernel-level)."""

    def __init__(self, max_m, max_n, max_k):
        self.h = _VP()
        st = lib().nitro_gemm_create(int(max_m), int(max_n), int(max_k), ctypes.byref(self.h))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_gemm_create")

    def run(self, a, b, c, stream=None):
        m, k = a.shape
        n = b.shape[0]
        st = lib().nitro_gemm_run(self.h, _ptr(a), _ptr(b), int(m), int(n), int(k), _ptr(c),
                                  _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_gemm_run")
        return c

    def status(self):
        return lib().nitro_gemm_status(self.h)

    def close(self):
        if getattr(self, "h", None):
            lib().nitro_gemm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class IntPrep:
    """Integer data pre-processing (App. A): fit mu / omega on a uint8 device
    tensor, then map uint8 tensors to int8 x_hat with them."""

    def __init__(self):
        self.h = _VP()
        st = lib().nitro_prep_create(ctypes.byref(self.h))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_prep_create")

    def fit(self, x, stream=None):
        st = lib().nitro_prep_fit(self.h, _ptr(x), int(x.numel()), _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_prep_fit")

    def apply(self, x, out, stream=None):
        if out.numel() != x.numel():
            raise ValueError("out must have as many elements as x")
        st = lib().nitro_prep_apply(self.h, _ptr(x), int(x.numel()), _ptr(out), _stream_ptr(stream))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_prep_apply")
        return out

    def stats(self):
        mu, om = ctypes.c_int64(), ctypes.c_int64()
        st = lib().nitro_prep_stats(self.h, ctypes.byref(mu), ctypes.byref(om))
        if st != NITRO_OK:
            raise NitroError(st, "nitro_prep_stats")
        return mu.value, om.value

    def close(self):
        if getattr(self, "h", None):
            lib().nitro_prep_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
