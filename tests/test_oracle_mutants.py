"""The pins must catch a wrong oracle.  Each case compiles a copy of
oracle/mc_oracle.c with one plausible slip planted (a dropped term, a wrong sign
or index, a transposed operand, a swapped slot, a wrong tie-break, a non-strict
threshold, ...) and runs the pin and worked-example tests against that build
(MC_ORACLE_SO); at least one of them must fail.  The mistakes are planted in the
oracle, on the CPU; no GPU is involved."""
import concurrent.futures as cf
import os
import subprocess
import sys
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "mc_oracle.c")

# (name, text in mc_oracle.c, replacement, which occurrence: 0 = first, -1 = every)
MUTANTS = [
    ("dequant: zero point dropped", "return (q - z) * s;", "return q * s;", 0),
    ("dequant: group of the wrong column", "int gi = k / m->group;", "int gi = (k + 1) % ng;", 0),
    ("expert: silu with the sign of the exponent flipped", "exp(-g)", "exp(g)", 0),
    ("expert: W1 and W3 swapped", "mco_gemv(w1, x, a1);\n    mco_gemv(w3, x, a3);",
     "mco_gemv(w3, x, a1);\n    mco_gemv(w1, x, a3);", 0),
    ("expert: down projection with W1", "mco_gemv(w2, a1, out);", "mco_gemv(w1, a1, out);", 0),
    ("routing: ties to the higher index", "if ((float)lt[e] > (float)lt[e0]) e0 = e;",
     "if ((float)lt[e] >= (float)lt[e0]) e0 = e;", 0),
    ("routing: no renormalisation", "double w0 = p0 / (p0 + p1);\n        double w1 = p1 / (p0 + p1);",
     "double w0 = p0;\n        double w1 = p1;", 0),
    ("ODP: non-strict threshold", "(w1 / w0 < mu)", "(w1 / w0 <= mu)", 0),
    ("ODP: primary keeps its weight when pruned", "if (prune) { w0 = 1.0; w1 = 0.0; }",
     "if (prune) { w1 = 0.0; }", 0),
    ("ODP: protection ignored", "int prune = (!prot) && (w1 / w0 < mu);", "int prune = (w1 / w0 < mu);", 0),
    ("drop: weights kept", "if (drop) { w0 = 0.0; w1 = 0.0; prune = 2; }", "if (drop) { prune = 2; }", 0),
    ("permutation: tokens descending", "for (int t = 0; t < T; ++t)\n            for (int slot = 0; slot < 2; ++slot) {",
     "for (int t = T - 1; t >= 0; --t)\n            for (int slot = 0; slot < 2; ++slot) {", 0),
    ("layer: primary slot skipped when pruned", "if ((slot == 1 && pruned[t]) || pruned[t] == 2) continue;",
     "if ((slot == 0 && pruned[t]) || pruned[t] == 2) continue;", -1),
    ("combine: routing weight dropped", "yt[h] += wt * eo[h];", "yt[h] += eo[h];", 0),
    ("rmsnorm: mean of squares not divided by H", "sqrt(ss / H + eps)", "sqrt(ss + eps)", 0),
]


def _mutate(src, old, new, which):
    assert old in src, old
    if which == -1:
        return src.replace(old, new)
    i = src.index(old)
    return src[:i] + new + src[i + len(old):]


def _run(case, tmp):
    name, old, new, which = case
    src = _mutate(open(SRC).read(), old, new, which)
    tag = "".join(c if c.isalnum() else "_" for c in name)
    c_path = os.path.join(tmp, tag + ".c")
    so_path = os.path.join(tmp, tag + ".so")
    with open(c_path, "w") as f:
        f.write(src)
    subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fno-fast-math", "-ffp-contract=off", "-o", so_path,
                           c_path, "-lm"])
    env = dict(os.environ, MC_ORACLE_SO=so_path)
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                        os.path.join(ROOT, "tests", "test_golden.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return name, r.returncode, r.stdout[-400:]


def test_every_planted_slip_fails_a_pin():
    with tempfile.TemporaryDirectory() as tmp:
        with cf.ThreadPoolExecutor(min(len(MUTANTS), os.cpu_count() or 2)) as ex:
            results = list(ex.map(lambda c: _run(c, tmp), MUTANTS))
    survivors = [(name, out) for name, rc, out in results if rc == 0]
    assert not survivors, "mutants no pin caught: %s" % [n for n, _ in survivors]
    # and the unmutated source passes the same tests
    assert all(rc != 0 for _, rc, _ in results)


def test_the_unmutated_oracle_passes_the_pins():
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                        os.path.join(ROOT, "tests", "test_golden.py")],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:]
