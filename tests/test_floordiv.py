"""Host-side pin of the library's division by invariant integers (the
multiply-high method of Granlund & Montgomery, PLDI 1994, Fig. 4.1) against
Python's exact floor and truncating division.  Compiles a host-only program
from the library header with nvcc; no GPU needed."""
import os
import random
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def divprog(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not available")
    d = tmp_path_factory.mktemp("div")
    src = d / "div.cu"
    src.write_text(r'''
#include <cstdio>
#include <cstdlib>
#include "nitro_internal.cuh"
int main() {
    unsigned long long dv; long long x;
    while (scanf("%llu %lld", &dv, &x) == 2) {
        nitro::FloorDiv f = nitro::FloorDiv::make(dv);
        long long f32 = 0;
        if (dv < (1ull << 32) && x >= -2147483648LL && x <= 2147483647LL)
            f32 = nitro::FloorDiv32::make((unsigned)dv).floor_div((int)x);
        printf("%lld %lld %lld\n", (long long)f.floor_div(x), (long long)f.trunc_div(x), f32);
    }
    return 0;
}
''')
    exe = d / "div"
    subprocess.run([nvcc, "-std=c++17", "-I", os.path.join(ROOT, "include"), "-I",
                    os.path.join(ROOT, "paper_2407_11698_gb300", "csrc"), str(src), "-o", str(exe)],
                   check=True, capture_output=True)
    return str(exe)


def test_floor_and_trunc_division_match_python(divprog):
    rnd = random.Random(5)
    ds = [1, 2, 3, 7, 10, 100, 256, 2304, 6912, 73728, 147456, 589824, 327680, 25000,
          9 * 512, 2**20 - 1, 2**31 - 1, 2**31, 2**32 + 1, 2**40 + 12345, 2**62 + 1]
    ds += [rnd.randrange(1, 2**63) for _ in range(40)]
    xs = [0, 1, -1, 2**63 - 1, -2**63, -2**63 + 1, 127, -127, -128, 2**31, -2**31 - 1,
          2**31 - 1, -2**31, -2**31 + 1]
    cases = []
    for d in ds:
        for x in xs + [rnd.randrange(-2**63, 2**63) for _ in range(60)] + \
                 [rnd.randrange(-4 * d, 4 * d) if d < 2**61 else 0 for _ in range(20)] + \
                 [rnd.randrange(-2**31, 2**31) for _ in range(30)] + \
                 [k * d + e for k in (-3, -1, 0, 1, 2) for e in (-1, 0, 1) if -2**63 <= k * d + e < 2**63]:
            cases.append((d, x))
    inp = "".join("%d %d\n" % c for c in cases)
    out = subprocess.run([divprog], input=inp, capture_output=True, text=True, check=True).stdout
    for (d, x), line in zip(cases, out.splitlines()):
        fl, tr, f32 = map(int, line.split())
        assert fl == x // d, (d, x)
        if d < 2**32 and -2**31 <= x < 2**31:
            assert f32 == x // d, ("32-bit", d, x)
        q = abs(x) // d
        assert tr == (q if x >= 0 else -q), (d, x)
