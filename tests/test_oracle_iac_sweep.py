"""Every single-token change of the IAC oracle's arithmetic fails a pin (CPU, a few seconds).

Each change below is planted, one at a time, in an in-memory copy of oracle/iac_oracle.py (as
tests/test_oracle_iac_mutants.py does for its hand-picked mistakes), and the copy must fail at least
one check of tests/test_oracle_iac.py. The changes are applied at every occurrence in the code
(docstrings and comments excluded): + and -, / and *, the constants 2.0, 1.0 and 0.0, min and max,
a dropped abs, sqrt or relu, == and !=, the start of the first per-job block, the offsets of the
pairwise features, and a dropped transpose."""

import numpy as np
import pytest

from tests import test_oracle_iac as pins
from tests import test_oracle_iac_mutants as M

OPS = [(" + ", " - "), (" - ", " + "), (" / ", " * "), (" * ", " / "), ("2.0", "1.0"), ("1.0", "0.0"),
       ("0.0", "1.0"), ("min(", "max("), ("max(", "min("), ("abs(", "("), (" == ", " != "), ("[0:", "[1:"),
       ("+ 1]", "]"), ("+ 2]", "+ 1]"), ("+ 3]", "+ 2]"), (".T", ""), ("np.sqrt(", "("), ("relu(", "(")]


def code_lines(lines):
    """Indices of the lines holding code: after the module docstring, outside docstrings and comments."""
    in_doc = False
    start = next(i for i, ln in enumerate(lines) if ln.startswith(("import", "from")))
    for i, ln in enumerate(lines):
        st = ln.strip()
        if i < start:
            continue
        if st.count('"""') == 1:
            in_doc = not in_doc
            continue
        if in_doc or '"""' in st or st.startswith("#") or not st:
            continue
        yield i


def mutants():
    lines = open(M.SRC).read().split("\n")
    out = []
    for i in code_lines(lines):
        ln = lines[i].split("#")[0]
        for a, b in OPS:
            at = ln.find(a)
            while at >= 0:
                out.append((i, a, b, "\n".join(lines[:i] + [ln[:at] + b + ln[at + len(a):]] + lines[i + 1:])))
                at = ln.find(a, at + 1)
    return out


def test_sweep_is_not_empty():
    assert len(mutants()) >= 40


def test_every_single_token_mutant_fails_a_pin():
    survivors = []
    for n, (i, a, b, src) in enumerate(mutants()):
        try:
            mod = M.module_from(src, f"iac_oracle_sweep_{n}")
        except Exception:
            continue                              # does not even load: caught
        caught = False
        with np.errstate(all="ignore"):
            for check in pins.CHECKS:
                try:
                    check(mod)
                except Exception:
                    caught = True
                    break
        if not caught:
            survivors.append(f"line {i + 1}: {a!r} -> {b!r}")
    assert not survivors, survivors
