"""Plant plausible mistakes in a copy of the oracle and require the pins to catch each.

The copy is compiled with gcc into a temporary directory; the committed
oracle is never modified.  Every mutant must fail at least one pin of
``oracle_pins`` -- otherwise the pins would not be able to tell that oracle
from a wrong one.
"""

import os
import subprocess

import pytest

import oracle as O
from tests import oracle_pins as P

pytestmark = pytest.mark.timeout(120)

SRC = os.path.join(os.path.dirname(O.__file__), "oracle.c")

# (name, original text, replacement) -- each original must occur exactly once.
MUTANTS = [
    ("drop the w(I(S)) term", "F[S] = best - wI[S];", "F[S] = best;"),
    ("ties keep the largest A", "if (c < best) { best = c; arg = A; }", "if (c <= best) { best = c; arg = A; }"),
    ("wrong complement operand", "int64_t c = F[A] + F[S ^ A];", "int64_t c = F[A] + F[S ^ low];"),
    ("skip the smallest split", "uint64_t sub = 0;\n  for (;;) {", "uint64_t sub = (0 - rest) & rest;\n  for (;;) {"),
    ("allow A = S", "if (sub == rest) break; /* A = S is not a split */",
     "if (sub == rest) { int64_t c = F[S] + F[0]; if (c < best) { best = c; arg = S; } break; }"),
    ("singleton base case 0", "F[S] = wI[S]; /* F({i}) = w(R_i) */", "F[S] = 0;"),
    ("union instead of intersection",
     "child[j] = I[j] & c->req[(int64_t)i * c->uw + j];", "child[j] = I[j] | c->req[(int64_t)i * c->uw + j];"),
    ("skipped subsets in the walk", "wi_visit(c, S | ((uint64_t)1 << i), i + 1, child, stack + c->uw);",
     "wi_visit(c, S | ((uint64_t)1 << i), i + 2, child, stack + c->uw);"),
    ("top layer never solved", "for (int k = 2; k <= m; ++k) {", "for (int k = 2; k < m; ++k) {"),
    ("single-subset weight over a union", "for (int64_t j = 0; j < words; ++j) acc[j] &= bits[(int64_t)i * words + j];",
     "for (int64_t j = 0; j < words; ++j) acc[j] |= bits[(int64_t)i * words + j];"),
    ("lowest bit taken wrong", "uint64_t low = S & (~S + 1);", "uint64_t low = S & (S - 1) ? S & (S - 1) & (~(S & (S - 1)) + 1) : S;"),
]


def _build_mutant(tmp_path, idx, old, new):
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation anchor not unique/found: {old!r}"
    text = text.replace(old, new)
    src = tmp_path / f"mutant{idx}.c"
    src.write_text(text)
    so = tmp_path / f"libmutant{idx}.so"
    subprocess.run(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=c11", str(src), "-o", str(so)], check=True,
                   timeout=120)
    return O.COracle(so)


@pytest.mark.parametrize("idx", range(len(MUTANTS)), ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, idx):
    name, old, new = MUTANTS[idx]
    C = _build_mutant(tmp_path, idx, old, new)
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(C)
        except Exception as e:  # an assertion, or a crash-free failure of any kind
            caught.append(pin.__name__)
            break
    assert caught, f"no pin detects the planted mistake: {name}"
