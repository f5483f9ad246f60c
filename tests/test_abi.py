"""Host-side checks of the C-ABI library (no GPU needed).

Builds libnitro.so if needed (cross-compiling needs no GPU), loads it, and
checks that every function include/*.h declares is exported, and that
argument checks that run before any device call reject bad input.
"""
import ctypes
import glob
import os
import re
import subprocess

import pytest

from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import build as nbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*[A-Za-z_][\w\s\*]*?\b(nitro_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    nbuild.build()
    return nb.lib()


def test_header_declares_the_four_step_entry_points():
    names = _declared_functions()
    for fn in ("nitro_init_block", "nitro_block_forward", "nitro_block_backward",
               "nitro_integersgd_step"):
        assert fn in names


def test_every_declared_symbol_is_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", nbuild.LIB], capture_output=True,
                         text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    missing = [n for n in _declared_functions() if n not in exported]
    assert not missing, missing
    for n in _declared_functions():
        assert hasattr(lib, n)


def test_status_strings(lib):
    assert nb.status_str(nb.NITRO_OK) == "ok"
    assert nb.status_str(nb.NITRO_ERR_OVERFLOW) == "integer overflow"
    assert nb.status_str(99) == "unknown status"


def _bad(**kw):
    base = dict(layers=[(nb.NITRO_CONV3X3, 1, 4, 6, 6, 1)], in_features=36, max_batch=2)
    base.update(kw)
    layers = base.pop("layers")
    in_f = base.pop("in_features")
    d, keep = nb.make_block_desc(layers, in_f, **base)
    st, h = nb.nitro_init_block(d, 1, None)
    return st, h, keep


@pytest.mark.parametrize("kw", [
    dict(alpha_inv=1),                                      # int8 output range needs alpha_inv >= 2
    dict(num_classes=0),
    dict(gamma_inv_lr=0),
    dict(eta_inv_fw=-1),
    dict(sgd_round=2),
    dict(max_batch=-1),
    dict(in_features=35),                                   # chain mismatch
    dict(layers=[(nb.NITRO_LINEAR, 36, 4, 2, 1, 0)]),       # linear takes h = w = 1
    dict(layers=[(nb.NITRO_LINEAR, 36, 4, 1, 1, 1)]),       # no pool after linear
    dict(layers=[(7, 1, 4, 6, 6, 0)]),                      # unknown kind
    dict(layers=[(nb.NITRO_CONV3X3, 1, 4, 6, 6, 1), (nb.NITRO_LINEAR, 37, 3, 1, 1, 0)]),
    dict(layers=[], in_features=0),
    dict(d_lr=-1),                                          # learning-layer input size
    dict(dropout_p16=-1),
    dict(dropout_p16=65537),                                # rate above 1
])
def test_init_rejects_bad_descriptors(lib, kw):
    st, h, _ = _bad(**kw)
    assert st == nb.NITRO_ERR_ARG and not h.value


def test_init_rejects_learning_pool_windows_above_a_byte(lib):
    # a 64 x 64 single-channel map brought to one feature needs a 64 x 64
    # window: its argmax no longer fits the byte the library stores it in
    st, h, _ = _bad(layers=[(nb.NITRO_CONV3X3, 1, 1, 64, 64, 0)], in_features=64 * 64, d_lr=1)
    assert st == nb.NITRO_ERR_UNSUPPORTED and not h.value


def test_null_handle_calls_are_rejected(lib):
    assert lib.nitro_block_set_dropout(None, 0) == nb.NITRO_ERR_ARG
    assert nb.nitro_block_forward(None, None, 0, None) == nb.NITRO_ERR_ARG
    assert nb.nitro_block_backward(None, None, None, 0, None) == nb.NITRO_ERR_ARG
    assert nb.nitro_integersgd_step(None) == nb.NITRO_ERR_ARG
    assert lib.nitro_block_set_hyper(None, 512, 0, 0) == nb.NITRO_ERR_ARG
    assert nb.nitro_block_status(None) == nb.NITRO_ERR_ARG
    nb.nitro_destroy_block(None)
    st, _ = nb.nitro_block_tensor_bytes(None, nb.NITRO_T_W, 0)
    assert st == nb.NITRO_ERR_ARG
    # the entry points added for the folded update, the data-parallel exchange
    # and the bounded-wait check reject a null handle before any device work
    assert nb.nitro_block_backward_update(None, None, None, 0, None) == nb.NITRO_ERR_ARG
    p, n = ctypes.c_void_p(), ctypes.c_size_t()
    assert lib.nitro_block_grad_device(None, nb.NITRO_T_DW, 0, ctypes.byref(p),
                                       ctypes.byref(n)) == nb.NITRO_ERR_ARG
    assert lib.nitro_block_diag_timeout(None, 1000, None) == nb.NITRO_ERR_ARG


def test_prep_null_handle_and_bad_sizes_are_rejected(lib):
    mu, om = ctypes.c_int64(), ctypes.c_int64()
    x = ctypes.c_void_p(16)            # never dereferenced: the checks come first
    assert lib.nitro_prep_fit(None, x, 10, None) == nb.NITRO_ERR_ARG
    assert lib.nitro_prep_apply(None, x, 10, x, None) == nb.NITRO_ERR_ARG
    assert lib.nitro_prep_stats(None, ctypes.byref(mu), ctypes.byref(om)) == nb.NITRO_ERR_ARG
    assert lib.nitro_prep_create(None) == nb.NITRO_ERR_ARG
    lib.nitro_prep_destroy(None)


def test_oracle_library_builds_independently():
    from oracle import build as obuild
    path = obuild.build()
    lib_o = ctypes.CDLL(path)
    assert hasattr(lib_o, "nor_conv3x3_fwd")
    # the oracle and the GPU library share no symbols
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True,
                         check=True).stdout
    assert not any(" nitro_" in l for l in out.splitlines())


def test_binding_structs_match_the_header(tmp_path):
    # sizes and field offsets of the C structs, as a C compiler lays them out
    # from include/nitro.h, against the binding's ctypes mirrors
    import shutil
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc:
        pytest.skip("no C compiler")
    fields = {
        "nitro_layer_desc": [f for f, _ in nb.nitro_layer_desc._fields_],
        "nitro_block_desc": [f for f, _ in nb.nitro_block_desc._fields_],
    }
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "nitro.h"', "int main(void) {"]
    for st, fs in fields.items():
        src.append('printf("%%s size %%zu\\n", "%s", sizeof(%s));' % (st, st))
        for f in fs:
            src.append('printf("%%s %%s %%zu\\n", "%s", "%s", offsetof(%s, %s));' % (st, f, st, f))
    src += ["return 0;", "}"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = {}
    for line in out:
        parts = line.split()
        if len(parts) == 3:
            got[(parts[0], parts[1])] = int(parts[2])
    for st, fs in fields.items():
        cls = getattr(nb, st)
        assert got[(st, "size")] == ctypes.sizeof(cls), st
        for f in fs:
            assert got[(st, f)] == getattr(cls, f).offset, (st, f)


def test_binding_constants_match_the_header(tmp_path):
    # every enum value and status bit the binding mirrors, from the header
    import shutil
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc:
        pytest.skip("no C compiler")
    names = [n for n in dir(nb) if n.startswith("NITRO_")]
    bits = {"STATUS_BIT_OVERFLOW": "NITRO_STATUS_BIT_OVERFLOW",
            "STATUS_BIT_BAD_LABEL": "NITRO_STATUS_BIT_BAD_LABEL",
            "STATUS_BIT_TIMEOUT": "NITRO_STATUS_BIT_TIMEOUT"}
    src = ["#include <stdio.h>", '#include "nitro.h"', "int main(void) {"]
    for n in names:
        src.append('printf("%s %%lld\\n", (long long)%s);' % (n, n))
    for py, c in bits.items():
        src.append('printf("%s %%lld\\n", (long long)%s);' % (py, c))
    src += ["return 0;", "}"]
    c = tmp_path / "consts.c"
    c.write_text("\n".join(src) + "\n")
    exe = tmp_path / "consts"
    subprocess.run([cc, "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    got = dict((l.split()[0], int(l.split()[1])) for l in out.splitlines() if l.strip())
    assert len(names) >= 26          # statuses, kinds, rounding, contractions, 13 tensors
    for n in names + list(bits):
        assert got[n] == getattr(nb, n), n


def test_product_package_never_reaches_the_oracle():
    # the library and its binding share nothing with the oracle: no Python
    # import of it, no include of its C file, no mention of its library
    pkg = os.path.join(ROOT, "paper_2407_11698_gb300")
    offenders = []
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if not fn.endswith((".py", ".cu", ".cuh", ".h", ".c", ".cpp")):
                continue
            path = os.path.join(dirpath, fn)
            text = open(path, encoding="utf-8").read()
            if re.search(r"^\s*(import oracle|from oracle\b)", text, flags=re.M) or \
                    "nitro_oracle" in text or "libnitro_oracle" in text:
                offenders.append(os.path.relpath(path, ROOT))
    assert not offenders, offenders
