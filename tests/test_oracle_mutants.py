"""The oracle's pins catch plausible mistakes in it.  Each case plants one
mistake (a dropped term, a wrong sign, a transposed operand, an index off by
one) in a copy of oracle/mosa_oracle.c, points the oracle at the copy and runs
the pin suite, which must fail.  The unmodified copy must pass."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "mosa_oracle.c")

# (what the mistake is, source text, replacement, replace every occurrence)
MUTANTS = [
    ("router sigmoid of -x", "return 1.0 / (1.0 + exp(-x));", "return 1.0 / (1.0 + exp(x));", False),
    ("TopK ties to the higher index", "return (a->t < b->t) ? -1 : (a->t > b->t);",
     "return (a->t > b->t) ? -1 : (a->t < b->t);", False),
    ("first token: rest not shifted back to token indices", "I[i] += 1;", "I[i] += 0;", False),
    ("mask without the diagonal", "if (I[i] < I[j]) return 0;", "if (I[i] <= I[j]) return 0;",
     False),
    ("mask reversed", "if (I[i] < I[j]) return 0;", "if (I[i] > I[j]) return 0;", False),
    ("local blocks off by one", "I[i] / window == I[j] / window",
     "(I[i] + 1) / window == I[j] / window", False),
    ("scale 1/h' instead of 1/sqrt(h')", "1.0 / sqrt((double)hp)", "1.0 / (double)hp", True),
    ("Y without the router scaling", "+= rs[i] * s.AWo[IDX2(i, c, d)];",
     "+= s.AWo[IDX2(i, c, d)];", False),
    ("dW_o without the router scaling", "acc += rs[i] * s.A[IDX2(i, p, hp)] * dXo",
     "acc += s.A[IDX2(i, p, hp)] * dXo", False),
    ("dA without the router scaling", "dA[IDX2(i, p, hp)] = rs[i] * acc;",
     "dA[IDX2(i, p, hp)] = acc;", False),
    ("dV from P untransposed", "acc += s.P[IDX2(i, j, k)] * dA[IDX2(i, p, hp)];",
     "acc += s.P[IDX2(j, i, k)] * dA[IDX2(i, p, hp)];", False),
    ("softmax backward without the row sum", "rowsum += s.P[IDX2(i, j, k)] * dp;",
     "rowsum += 0.0 * dp;", False),
    ("dK from dS untransposed", "ak += dS[IDX2(j, i, k)] * s.Q[IDX2(j, p, hp)];",
     "ak += dS[IDX2(i, j, k)] * s.Q[IDX2(j, p, hp)];", False),
    ("dQ without the 1/sqrt(h') scale", "dQ[IDX2(i, p, hp)] = aq * scale;",
     "dQ[IDX2(i, p, hp)] = aq;", False),
    ("router gradient without sigma'", "dr[i] * rs[i] * (1.0 - rs[i])", "dr[i] * rs[i]", False),
    ("dX without the router term", "double acc = unit_scores ? 0.0 : dlogit[i] * Wr[IDX2(c, h, H)];",
     "double acc = 0.0;", False),
    ("RoPE frequencies over h' instead of h'/2", "-2.0 * p / (double)half", "-2.0 * p / (double)hp",
     False),
    ("RoPE not a rotation", "v[2 * p] = x0 * c - x1 * sn;", "v[2 * p] = x0 * c + x1 * sn;", False),
    ("RoPE gradient of dQ turned forward", "rope_rotate(dQ + IDX2(i, 0, hp), hp, Ibh[i], -1);",
     "rope_rotate(dQ + IDX2(i, 0, hp), hp, Ibh[i], +1);", False),
]


def run_pins(src_path):
    env = dict(os.environ, MOSA_ORACLE_SRC=src_path)
    return subprocess.run([sys.executable, "-m", "pytest", os.path.join(ROOT, "tests",
                                                                        "test_oracle_pins.py"),
                           "-x", "-q", "-p", "no:cacheprovider"],
                          cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)


def test_unmodified_copy_passes(tmp_path):
    path = tmp_path / "oracle_copy.c"
    path.write_text(open(SRC).read())
    out = run_pins(str(path))
    assert out.returncode == 0, out.stdout[-3000:]


@pytest.mark.parametrize("what,old,new,every", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_the_pins(tmp_path, what, old, new, every):
    text = open(SRC).read()
    n = text.count(old)
    assert n == 1 or (every and n > 1), f"{what}: the source text moved ({n} matches)"
    path = tmp_path / "mutant.c"
    path.write_text(text.replace(old, new))
    so = tmp_path / "mutant_check.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-o", str(so),
                    str(path), "-lm"], check=True)             # the mutant compiles
    out = run_pins(str(path))
    assert out.returncode == 1, f"{what}: pins passed\n" + out.stdout[-2000:]
