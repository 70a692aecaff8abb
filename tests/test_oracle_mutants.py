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
    # block maximum, exponent range, special values, exact summation
    "block maximum without the absolute value": ("else if (fabs(x[i]) > amax) amax = fabs(x[i]);",
                                                 "else if (x[i] > amax) amax = x[i];"),
    "exponent floor at -120": ("if (E < -127) E = -127;", "if (E < -120) E = -120;"),
    "scale byte 255 read as a number": ("if (scale == 255) return NAN;", "if (scale == 256) return NAN;"),
    "activation scales in block order": ("pscales[r * nb + s] = scales[r * nb + kb];",
                                         "pscales[r * nb + s] = scales[r * nb + s];"),
    "bf16 NaN block written as Inf": ("S == 255 ? 0x7FC0 :", "S == 255 ? 0x7F80 :"),
    "two-sum low part with the wrong sign": ("double lo = y - (hi - x);", "double lo = (hi - x) - y;"),
    "exact sum without the half-way fix": ("if (y == x - hi) hi = x;", "if (0) hi = x;"),
    "e4m3 subnormal scale": ("double k = ldexp(a, 9);", "double k = ldexp(a, 8);"),
    "4-bit weight sign in bit 2": ("const uint8_t nib = (uint8_t)(((c[e] < 0) << 3) | mag);",
                                   "const uint8_t nib = (uint8_t)(((c[e] < 0) << 2) | mag);"),
    "4-bit weight nibbles swapped": ("*byte |= (uint8_t)(within < 4 ? nib : (nib << 4));",
                                     "*byte |= (uint8_t)(within < 4 ? (nib << 4) : nib);"),
    "6/8-bit weight scale on the next row": ("slot[4096 + rr] = scales[r * nb + kb];",
                                             "slot[4096 + (rr + 1) % 128] = scales[r * nb + kb];"),
    "4-bit plane elements reversed": ("planes[r * kp + 32 * s + i] = (uint8_t)ch;",
                                      "planes[r * kp + 32 * s + (31 - i)] = (uint8_t)ch;"),
    "bf16 plane low byte from the high": ("planes[r * kp + p68 + 64 * (s - n4) + 2 * i] = (uint8_t)(v & 0xFF);",
                                          "planes[r * kp + p68 + 64 * (s - n4) + 2 * i] = (uint8_t)((v >> 8) & 0xFF);"),
    "6/8-bit scale tile slots swapped": ("int64_t j = 2 * (st - st4) + q;", "int64_t j = 2 * (st - st4) + 1 - q;"),
    "ties away by floor(v + 1/2)": ("? round(v) : nearbyint(v)", "? floor(v + 0.5) : nearbyint(v)"),
    "error bound from signed terms": ("for (int64_t kb = 0; kb < nb; ++kb) terms[kb] = fabs(terms[kb]);",
                                      "for (int64_t kb = 0; kb < nb; ++kb) terms[kb] = terms[kb];"),
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


def _c_pins(tmp_path, name, old, new):
    d = tmp_path / name.replace(" ", "_").replace("/", "-")
    d.mkdir()
    env = dict(os.environ, MXO_LIB=_build(d, name, old, new), OMP_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return name, r


def test_pins_reject_every_planted_mistake(tmp_path):
    """Each altered copy must make some pin fail (pytest's return code 1; 0
    would mean the mistake went unseen, other codes are errors of the run)."""
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(max(1, min(8, os.cpu_count() or 1))) as ex:
        runs = list(ex.map(lambda kv: _c_pins(tmp_path, kv[0], *kv[1]), MUTANTS.items()))
    unseen = [f"{name}: {r.returncode}\n{r.stdout[-600:]}" for name, r in runs if r.returncode != 1]
    assert not unseen, "\n".join(unseen)


def test_the_unaltered_oracle_passes_the_same_run(tmp_path):
    lib = _build(tmp_path, "none", "ldexp((double)d, ea + ew)", "ldexp((double)d, ea + ew)")
    env = dict(os.environ, MXO_LIB=lib, OMP_NUM_THREADS="2")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:]


# ------------------------------------------------- the Python oracles
PY_MUTANTS = {
    # oracle/alloc.py (Alg. 1, Theorem 1, Alg. 3), pinned by test_oracle_alloc.py
    "sensitivity as a sum of |x|": ("oracle/alloc.py", "return np.sum(x * x, axis=0)",
                                    "return np.sum(np.abs(x), axis=0)"),
    "R without the 8-bit columns": ("oracle/alloc.py", "num = (B - 4.0) * d.sum() - 4.0 * BLOCK * n",
                                    "num = (B - 4.0) * d.sum()"),
    "R with the 6-bit gain halved": ("oracle/alloc.py", "den = np.sum(2.0 * s * (d - BLOCK))",
                                     "den = np.sum(s * (d - BLOCK))"),
    "N6 rounded": ("oracle/alloc.py", "v = math.floor(R * s_layer * (d_in - BLOCK))",
                   "v = round(R * s_layer * (d_in - BLOCK))"),
    "N6 unclamped": ("oracle/alloc.py", "return int(min(max(v, 0), d_in - BLOCK))", "return int(max(v, 0))"),
    "ties in reverse order": ("oracle/alloc.py", 'np.argsort(-s, kind="stable")',
                              'np.argsort(s, kind="stable")[::-1]'),
    "no 8-bit block": ("oracle/alloc.py", "bits[0] = 8", "bits[0] = 6"),
    "bf16 decoded one bit off": ("oracle/alloc.py", "astype(np.uint32) << 16", "astype(np.uint32) << 15"),
    "average width per block": ("oracle/alloc.py", "* BLOCK for b in bits_per_layer", "for b in bits_per_layer"),
    "one 6-bit block too many": ("oracle/alloc.py", "bits[1:1 + n6b] = 6", "bits[1:2 + n6b] = 6"),
    # oracle/attention.py (KV cache, Appendix A.2), pinned by test_oracle_attention.py
    "query head reads the wrong KV head": ("oracle/attention.py", "c = (h // G) * D", "c = (h % n_kv_heads) * D"),
    "scores without the scale": ("oracle/attention.py", "s = scale * (kh @ q[h])", "s = kh @ q[h]"),
    "weights not normalised": ("oracle/attention.py", "out[h] = (p @ vh) / np.sum(p)", "out[h] = (p @ vh)"),
    "sequence rows at the wrong place": ("oracle/attention.py", "rows = slice(b * T_cap, b * T_cap + T)",
                                         "rows = slice(b * T, b * T + T)"),
    "cache values on the 8-bit grid": ("oracle/attention.py", "return mxo.dequantize(codes, scales, bits)",
                                       "return mxo.dequantize(codes, scales, np.full(len(bits), 8, np.uint8))"),
    "scores against the value cache": ("oracle/attention.py", "s = scale * (kh @ q[h])", "s = scale * (vh @ q[h])"),
    "sequence lengths ignored": ("oracle/attention.py", "T = int(lengths[b])", "T = T_cap"),
    "an empty sequence not read as zeros": ("oracle/attention.py", "if T > 0:", "if T >= 0:"),
}
PINS = {"oracle/alloc.py": "test_oracle_alloc.py", "oracle/attention.py": "test_oracle_attention.py"}


def _py_tree(tmp_path, rel, old, new):
    """A copy of tests/ and oracle/ with one oracle file altered (the package
    linked): the copied conftest puts this tree first on the path."""
    import shutil
    skip = shutil.ignore_patterns("__pycache__", "_build")
    shutil.copytree(os.path.join(ROOT, "tests"), tmp_path / "tests", ignore=skip)
    shutil.copytree(os.path.join(ROOT, "oracle"), tmp_path / "oracle", ignore=skip)
    os.symlink(os.path.join(ROOT, "paper_2607_17733_gb300"), tmp_path / "paper_2607_17733_gb300")
    f = tmp_path / rel
    src = f.read_text()
    assert src.count(old) == 1, f"the text to alter must occur once in {rel}"
    f.write_text(src.replace(old, new))
    return tmp_path


def _run_pins(tree, rel):
    from oracle import mxo
    env = dict(os.environ, MXO_LIB=mxo.build(), OMP_NUM_THREADS="1")  # the C oracle as built
    return subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                           str(tree / "tests" / PINS[rel])],
                          cwd=str(tree), env=env, capture_output=True, text=True, timeout=600)


def test_python_pins_reject_every_planted_mistake(tmp_path):
    from concurrent.futures import ThreadPoolExecutor

    def one(item):
        name, (rel, old, new) = item
        d = tmp_path / name.replace(" ", "_")
        d.mkdir()
        return name, _run_pins(_py_tree(d, rel, old, new), rel)

    with ThreadPoolExecutor(max(1, min(8, os.cpu_count() or 1))) as ex:
        runs = list(ex.map(one, PY_MUTANTS.items()))
    unseen = [f"{name}: {r.returncode}\n{r.stdout[-600:]}" for name, r in runs if r.returncode != 1]
    assert not unseen, "\n".join(unseen)


@pytest.mark.parametrize("rel", list(PINS))
def test_the_unaltered_python_oracles_pass_the_same_run(tmp_path, rel):
    r = _run_pins(_py_tree(tmp_path, rel, "import numpy as np", "import numpy as np"), rel)
    assert r.returncode == 0, r.stdout[-2000:]
