"""Planted mistakes in the oracle (on the CPU): each copy of oracle/mxo.c
below carries one plausible error -- in the arithmetic (an exponent off by
one, ties to the wrong side, a clamp that admits -2^(b-1), a grid one
fraction bit off, a dropped or misaligned element in the block dot, a scale
with the wrong sign, a NaN of one operand ignored, a naive sum) or in the
storage formats and MMA operands (nibble order, word layout, sign bit, scale
byte place, width-group order, the e4m3 and bf16 encoders, plane digits, the
scale-tile layout) -- and is built into its own library.  (Where the
digits of a 6/8-bit code split is not pinned: any exact split is as good,
and no kernel reads the digit form; the bf16 form is their operand.)  The oracle's pins (tests/test_oracle_pins.py, run against that
library) must reject every copy: this is what lets the pins vouch for the
oracle."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "mxo.c")

MUTANTS = {
    "exponent off by one": ("frexp(amax, &e);\n        E = e - 1;", "frexp(amax, &e);\n        E = e;"),
    "ties to the wrong side": ("(rounding == MXO_RHAZ) ? round(v) : nearbyint(v)",
                               "(rounding == MXO_RHAZ) ? nearbyint(v) : round(v)"),
    "clamp admits -2^(b-1)": ("if (r < -Q) r = -Q;", "if (r < -Q - 1) r = -Q - 1;"),
    "grid one fraction bit off": ("ldexp(x[i], (b - 2) - E)", "ldexp(x[i], (b - 1) - E)"),
    "value of a code one bit off": ("return ldexp((double)m, (int)scale - 127 - (b - 2));",
                                    "return ldexp((double)m, (int)scale - 127 - (b - 1));"),
    "an element dropped from the block dot": ("for (int i = 0; i < MXO_BLOCK; ++i)\n            d +=",
                                              "for (int i = 1; i < MXO_BLOCK; ++i)\n            d +="),
    "weight elements in reverse order": ("* (int64_t)wc[kb * MXO_BLOCK + i];",
                                         "* (int64_t)wc[kb * MXO_BLOCK + (MXO_BLOCK - 1 - i)];"),
    "weight scale with the wrong sign": ("ldexp((double)d, ea + ew)", "ldexp((double)d, ea - ew)"),
    "a NaN weight block ignored": ("if (as[kb] == 255 || ws[kb] == 255) nan = 1;", "if (as[kb] == 255) nan = 1;"),
    "naive summation": ("*y = mxo_fsum(terms, nb);",
                        "{ double s_ = 0; for (int64_t q_ = 0; q_ < nb; ++q_) s_ += terms[q_]; *y = s_; }"),
    # storage formats and MMA operands (every altered copy writes inside its buffers)
    "activation nibbles swapped": ("(i % 2) ? (nib << 4) : nib", "(i % 2) ? nib : (nib << 4)"),
    "weight nibble word layout": ("4 * i + (within % 4)", "4 * i + (within / 2)"),
    "6/8-bit weight sign in bit 6": ("(uint8_t)(((c[e] < 0) << 7) | mag)", "(uint8_t)(((c[e] < 0) << 6) | mag)"),
    "4-bit weight scale byte one place early": ("slot[2048 + rr]", "slot[2047 + rr]"),
    "8-bit group before the 6-bit group": ("const int widths[3] = {4, 6, 8};", "const int widths[3] = {4, 8, 6};"),
    "e4m3 exponent bias": ("code = ((E + 7) << 3) | (int)k;", "code = ((E + 6) << 3) | (int)k;"),
    "bf16 subnormal scale": ("double k = ldexp(a, 133);", "double k = ldexp(a, 132);"),
    "4-bit plane digit m/2": ("if (b == 4) { *hi = m / 4.0;", "if (b == 4) { *hi = m / 2.0;"),
    "low digit one bit off": ("*lo = ldexp((double)l, -(b - 2));", "*lo = ldexp((double)l, -(b - 1));"),
    "scale tile transposed": ("* 16 + w * 4 + q] = scales", "* 16 + q * 4 + w] = scales"),
}


def _build(tmp_path, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"{name}: the text to alter must occur once in mxo.c"
    path = tmp_path / "mxo.c"
    path.write_text(src.replace(old, new))
    lib = tmp_path / "libmxo_mutant.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
                    "-ffp-contract=off", str(path), "-o", str(lib), "-lm"], check=True)
    return str(lib)


@pytest.mark.parametrize("name", list(MUTANTS))
def test_pins_reject_a_planted_mistake(tmp_path, name):
    lib = _build(tmp_path, name, *MUTANTS[name])
    env = dict(os.environ, MXO_LIB=lib, OMP_NUM_THREADS="2")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    # 1: some pin failed (0 would mean the mistake went unseen; other codes are
    # errors of the run itself)
    assert r.returncode == 1, f"{name}: pins returned {r.returncode}\n{r.stdout[-2000:]}"


def test_the_unaltered_oracle_passes_the_same_run(tmp_path):
    lib = _build(tmp_path, "none", "ldexp((double)d, ea + ew)", "ldexp((double)d, ea + ew)")
    env = dict(os.environ, MXO_LIB=lib, OMP_NUM_THREADS="2")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:]
