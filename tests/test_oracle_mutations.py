"""The oracle's pins catch plausible mistakes (CPU only). Each case plants one
mistake in a scratch copy of the oracle's C sources, builds it, and runs the pin
suites against that build in a child process (the oracle loads the library named
by DC_ORACLE_LIB): at least one pin must fail. An unmutated copy must pass."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE = os.path.join(ROOT, "oracle")
SOURCES = ("dynacomm_oracle.c", "greedy_oracle.c", "dynacomm_oracle.h")
DP_PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")
GREEDY_PINS = os.path.join(ROOT, "tests", "test_greedy_pins.py")

# (name, file, text, planted text, pin suites that must catch it)
MUTATIONS = [
    ("forward pull count one short (n-1)*dt", "dynacomm_oracle.c",
     "return max64(before, (int64_t)n * dt + T[m]) + (C[m] - C[k]);",
     "return max64(before, (int64_t)(n - 1) * dt + T[m]) + (C[m] - C[k]);", (DP_PINS,)),
    ("backward push without its dt", "dynacomm_oracle.c",
     "return max64(before, C[m]) + dt + (T[m] - T[k]); /* Eq. 9 */",
     "return max64(before, C[m]) + (T[m] - T[k]); /* Eq. 9 */", (DP_PINS,)),
    ("split tie-break keeps the larger k", "dynacomm_oracle.c",
     "if (arg < 0 || c < best) {", "if (arg < 0 || c <= best) {", (DP_PINS,)),
    ("segment-count tie-break keeps the larger n", "dynacomm_oracle.c",
     "if (X[(size_t)n * W + (size_t)L] < X[(size_t)s * W + (size_t)L]) s = n;",
     "if (X[(size_t)n * W + (size_t)L] <= X[(size_t)s * W + (size_t)L]) s = n;", (DP_PINS,)),
    ("decision bit one layer off", "dynacomm_oracle.c",
     "if (k >= 1 && k <= L - 1) d[k] = 1;", "if (k >= 1 && k <= L - 2) d[k + 1] = 1;",
     (DP_PINS,)),
    ("backward prefix taken in forward order", "dynacomm_oracle.c",
     "S[m] = S[m - 1] + v[L - m];", "S[m] = S[m - 1] + v[m - 1];", (DP_PINS,)),
    ("replay forgets the pull's dt", "dynacomm_oracle.c",
     "int64_t xfer = dt;", "int64_t xfer = 0;", (DP_PINS,)),
    ("SplitMix64 mixer constant off by one", "dynacomm_oracle.c",
     "0xbf58476d1ce4e5b9ull", "0xbf58476d1ce4e5b8ull", (DP_PINS,)),
    ("floor instead of ceiling for costs", "dynacomm_oracle.c",
     "static int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }",
     "static int64_t ceil_div(int64_t a, int64_t b) { return a / b; }", (DP_PINS,)),
    ("log-uniform knots spaced j/511", "dynacomm_oracle.c",
     "double x = (double)j / 512.0;", "double x = (double)j / 511.0;", (DP_PINS,)),
    ("greedy least slack keeps the later tie", "greedy_oracle.c",
     "(pick < 0 || slack[c] < slack[pick])", "(pick < 0 || slack[c] <= slack[pick])",
     (GREEDY_PINS,)),
    ("greedy largest slack keeps the later tie", "greedy_oracle.c",
     "if (slack[c] > slack[pick]) pick = c;", "if (slack[c] >= slack[pick]) pick = c;",
     (GREEDY_PINS,)),
]


def _build(tmp, mutation=None):
    for f in SOURCES:
        shutil.copy(os.path.join(ORACLE, f), tmp)
    if mutation is not None:
        _, fname, text, planted, _ = mutation
        path = os.path.join(tmp, fname)
        src = open(path).read()
        assert src.count(text) == 1, f"mutation site not unique in {fname}: {text}"
        open(path, "w").write(src.replace(text, planted))
    lib = os.path.join(tmp, "liboracle_mut.so")
    subprocess.check_call(["gcc", "-std=gnu99", "-O2", "-fPIC", "-shared", "-w", "-o", lib,
                           os.path.join(tmp, "dynacomm_oracle.c"),
                           os.path.join(tmp, "greedy_oracle.c"), "-lm", "-lpthread"])
    return lib


def _pins_pass(lib, suites):
    env = dict(os.environ, DC_ORACLE_LIB=lib)
    res = subprocess.run([sys.executable, "-m", "pytest", *suites, "-x", "-q", "-m", "not gpu",
                          "-p", "no:cacheprovider"], cwd=ROOT, env=env, capture_output=True,
                         text=True, timeout=600)
    return res.returncode == 0, res.stdout[-2000:]


def test_unmutated_copy_passes(tmp_path):
    ok, out = _pins_pass(_build(str(tmp_path)), (DP_PINS, GREEDY_PINS))
    assert ok, out


@pytest.mark.parametrize("mutation", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_mutation(tmp_path, mutation):
    ok, out = _pins_pass(_build(str(tmp_path), mutation), mutation[4])
    assert not ok, f"no pin failed for the planted mistake: {mutation[0]}\n{out}"
