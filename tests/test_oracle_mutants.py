"""The oracle's pins catch plausible mistakes (CPU only).

Each case plants one mistake in a copy of oracle/oracle.c: a dropped term,
a wrong sign, index or operand, the other mask alignment or head mapping,
the wrong logarithm.  The copy is compiled on its own, and the pin tests of
test_oracle.py run against it in a child process.  At least one pin must
fail, or the process must die.  The unmodified source, built the same way,
passes every pin.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.c")

MUTANTS = [
    # (name, text in oracle.c, replacement)
    ("scale dropped", "x[j] = scale * dot;", "x[j] = dot;"),
    ("mask one key too many", "int64_t last = i + delta;", "int64_t last = i + delta + 1;"),
    ("mask one key too few", "int64_t last = i + delta;", "int64_t last = i + delta - 1;"),
    ("top-left mask alignment", "int64_t last = i + delta;", "int64_t last = i;"),
    ("interleaved head mapping", "int32_t g = h / G;", "int32_t g = h % Hkv;"),
    ("LSE without the max", "*lse = m + log(l);", "*lse = log(l);"),
    ("LSE in base 2", "*lse = m + log(l);", "*lse = m + log2(l);"),
    ("O not normalised", "o_row[c] /= l;", "o_row[c] /= 1.0;"),
    ("max not subtracted", "double p = exp(x[j] - m);", "double p = exp(x[j]);"),
    ("exponent sign flipped", "double p = exp(x[j] - m);", "double p = exp(m - x[j]);"),
    ("scores against V", "const uint16_t *krow = k + ", "const uint16_t *krow = v + "),
    ("values from K", "const uint16_t *vrow = v + ", "const uint16_t *vrow = k + "),
    ("query row of the kv head", "const uint16_t *qrow = q + (token * Hq + h)",
     "const uint16_t *qrow = q + (token * Hq + g)"),
    ("keys indexed by the query offsets", "const uint16_t *krow = k + ((cu_k[s] + j)",
     "const uint16_t *krow = k + ((cu_q[s] + j)"),
    ("empty row LSE zero", "*lse = -INFINITY;", "*lse = 0.0;"),
    ("bf16 widened with the wrong shift", "uint32_t u = (uint32_t)bits << 16;", "uint32_t u = (uint32_t)bits << 15;"),
]


def build_variant(text, path):
    with open(path.with_suffix(".c"), "w") as f:
        f.write(text)
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread", "-o", str(path),
                    str(path.with_suffix(".c")), "-lm"], check=True)


def run_pins(lib_path):
    env = dict(os.environ, OPATTN_ORACLE_LIBRARY=str(lib_path))
    return subprocess.run([sys.executable, "-m", "pytest", os.path.join("tests", "test_oracle.py"), "-x", "-q",
                           "-p", "no:cacheprovider"], cwd=ROOT, env=env, capture_output=True, text=True,
                          timeout=600)


def test_every_mutation_site_is_in_the_source():
    src = open(SRC).read()
    for name, old, _ in MUTANTS:
        assert src.count(old) == 1, name


def test_unmodified_copy_passes_every_pin(tmp_path):
    lib = tmp_path / "liboracle_copy.so"
    build_variant(open(SRC).read(), lib)
    r = run_pins(lib)
    assert r.returncode == 0, r.stdout[-3000:]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(name, old, new, tmp_path):
    lib = tmp_path / "liboracle_mutant.so"
    build_variant(open(SRC).read().replace(old, new, 1), lib)
    r = run_pins(lib)
    assert r.returncode != 0, f"no pin caught the mistake '{name}':\n{r.stdout[-2000:]}"
