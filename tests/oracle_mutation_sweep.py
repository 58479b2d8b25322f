"""Mutation sweep of the C oracle (test infrastructure, run by hand; about four minutes on one core).

Every single-token change of a comparison (< <= > >=), an arithmetic operator (+ - * /), a
compound assignment, the constant 0.0, an equality test or the 1-based update number is planted in
a temporary copy of oracle/esp_oracle.c. Each copy is compiled and runs the pin suite of
tests/test_oracle_mutants.py in a child process. Mutants that no pin catches are printed. They are
either equivalent to the original (the change only matters at an equality where both branches
give the same value, or for a sign of zero) or read or write out of bounds, which
tests/test_host_sanitized.py reports when it runs the same pins under AddressSanitizer.

    python -m tests.oracle_mutation_sweep [--sanitize-survivors]

With --sanitize-survivors every mutant that the pins miss is also run under the sanitizers, and the
first report (or its absence) is printed beneath it.
"""

from __future__ import annotations

import os
import shutil
import subprocess
import sys
import tempfile

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
OPS = [(" < ", " <= "), (" <= ", " < "), (" > ", " >= "), (" >= ", " > "), (" + ", " - "), (" - ", " + "),
       (" * ", " / "), ("+= ", "-= "), ("0.0", "1.0"), ("== ", "!= "), ("it + 1", "it")]


def candidates(lines):
    for i, ln in enumerate(lines):
        st = ln.strip()
        if not st or st.startswith(("/*", "*", "#", "//")):
            continue
        for a, b in OPS:
            at = ln.find(a)
            while at >= 0:
                yield i, ln[:at] + b + ln[at + len(a):]
                at = ln.find(a, at + 1)


def child(lib_path: str) -> int:
    import numpy as np

    import oracle
    from tests import test_oracle_mutants as mut
    lib = oracle.load(lib_path)
    with np.errstate(all="ignore"):
        try:
            failures = mut.failing_pins(lib)
        except Exception:
            failures = 1
    print("FAILING_PINS", failures)
    return 0


def main() -> int:
    if len(sys.argv) == 3 and sys.argv[1] == "--child":
        return child(sys.argv[2])
    sanitize = "--sanitize-survivors" in sys.argv
    sys.path.insert(0, ROOT)
    import oracle
    src_path = os.path.join(ROOT, "oracle", "esp_oracle.c")
    lines = open(src_path).read().split("\n")
    tmp = tempfile.mkdtemp()
    shutil.copy(os.path.join(ROOT, "oracle", "esp_oracle.h"), tmp)
    total = survivors = 0
    for n, (i, new_line) in enumerate(candidates(lines)):
        mutated = lines[:i] + [new_line] + lines[i + 1:]
        c, so = os.path.join(tmp, f"m{n}.c"), os.path.join(tmp, f"m{n}.so")
        open(c, "w").write("\n".join(mutated))
        if subprocess.run(["gcc", *oracle.CFLAGS, c, "-o", so, "-lm"], capture_output=True).returncode:
            continue
        total += 1
        try:
            r = subprocess.run([sys.executable, "-m", "tests.oracle_mutation_sweep", "--child", so], cwd=ROOT,
                               capture_output=True, text=True, timeout=120)
            caught = "FAILING_PINS 0" not in r.stdout
        except subprocess.TimeoutExpired:
            caught = True
        if not caught:
            survivors += 1
            print(f"not caught, line {i + 1}: {lines[i].strip()}  =>  {new_line.strip()}", flush=True)
            if sanitize:
                print("    sanitizers: " + sanitized_verdict(mutated, tmp, n), flush=True)
    shutil.rmtree(tmp, ignore_errors=True)
    print(f"{survivors} of {total} compiled mutants not caught by the pins")
    return 0


def sanitized_verdict(mutated_lines, tmp, n):
    """Runs the pins on the mutant built with AddressSanitizer and UndefinedBehaviorSanitizer (as
    tests/test_host_sanitized.py does) and returns the first report, or says there was none."""
    from tests import test_host_sanitized as san
    rt = san._runtime("libasan.so")
    if rt is None:
        return "unavailable (no AddressSanitizer runtime)"
    d = os.path.join(tmp, f"san{n}")
    os.makedirs(d, exist_ok=True)
    src = "\n".join(mutated_lines)
    c = os.path.join(d, "esp_oracle.c")
    open(c, "w").write(src)
    shutil.copy(os.path.join(ROOT, "oracle", "esp_oracle.h"), d)
    import oracle
    so = os.path.join(d, "liboracle_san.so")
    subprocess.check_call(["gcc", *oracle.CFLAGS, *san.SAN, c, "-o", so, "-lm"])
    r = san.run_child(rt, so, os.path.join(d, "out.npz"), pins=True)
    reports = [ln.strip() for ln in r.stderr.splitlines() if "ERROR: AddressSanitizer" in ln or "runtime error" in ln]
    if r.returncode != 0 and reports:
        return "reported: " + reports[0][:120]
    return "no report (equivalent to the original, or undetected)"


if __name__ == "__main__":
    sys.exit(main())
