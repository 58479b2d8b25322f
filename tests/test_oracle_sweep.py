"""Every single-token mutant of the C oracle fails a pin, is equivalent to the original, or is
reported by the sanitizers (CPU, about half a minute on 8 cores).

The mutants are those of tests/oracle_mutation_sweep.py: each comparison, arithmetic operator,
compound assignment, constant 0.0, equality test and update number of oracle/esp_oracle.c changed
in turn. Each compiles in a temporary directory, and the pin suite of tests/test_oracle_mutants.py
runs against it in a child process. The mutants that survive must be in the list below:
- **Equivalent.** The change matters only at an equality where both branches give the same value,
  only for the sign of a zero price, or only for an allocation size when a job count is zero.
- **One past the end.** A loop bound that reads one element past its array. These must also make
  the sanitized pin run of tests/test_host_sanitized.py fail.
A new survivor means a pin is missing."""

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys
import tempfile

import pytest

import oracle
from tests import oracle_mutation_sweep as sweep
from tests import test_host_sanitized as san

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (original line, mutated line), both stripped
EQUIVALENT = {
    ("lambda_out[k] = moved > 0.0 ? moved : 0.0; /* projection onto lambda >= 0 */",
     "lambda_out[k] = moved >= 0.0 ? moved : 0.0; /* projection onto lambda >= 0 */"),
    ("lambda_out[k] = moved > 0.0 ? moved : 0.0; /* projection onto lambda >= 0 */",
     "lambda_out[k] = moved > 0.0 ? moved : 0.0; /* projection onto lambda > 0 */"),
    ("int32_t *sel = (int32_t *)calloc((size_t)(J > 0 ? J : 1), sizeof(int32_t));",
     "int32_t *sel = (int32_t *)calloc((size_t)(J >= 0 ? J : 1), sizeof(int32_t));"),
    ("double *score = (double *)calloc((size_t)(J > 0 ? J : 1), sizeof(double));",
     "double *score = (double *)calloc((size_t)(J >= 0 ? J : 1), sizeof(double));"),
    ("if (g < best_dual)", "if (g <= best_dual)"),
    ("if (d > delta)", "if (d >= delta)"),
    ("if (fabs(lambda[k]) > scale)", "if (fabs(lambda[k]) >= scale)"),
    ("if (add > beta_max)", "if (add >= beta_max)"),
    ("if (excess < 0.0)", "if (excess <= 0.0)"),
    ("const double gamma = esp_oracle_penalty(c, cur, gamma0, s_hat ? alpha : 0.0, s_hat ? s_hat[o] : 0.0,",
     "const double gamma = esp_oracle_penalty(c, cur, gamma0, s_hat ? alpha : 1.0, s_hat ? s_hat[o] : 0.0,"),
    ("const double gamma = esp_oracle_penalty(c, cur, gamma0, s_hat ? alpha : 0.0, s_hat ? s_hat[o] : 0.0,",
     "const double gamma = esp_oracle_penalty(c, cur, gamma0, s_hat ? alpha : 0.0, s_hat ? s_hat[o] : 1.0,"),
    ("s_hat ? tau[j] : 0.0);", "s_hat ? tau[j] : 1.0);"),
    ("if (q_units[o * R + r] < m)", "if (q_units[o * R + r] <= m)"),
    ("if (c < 1)", "if (c <= 1)"),
}
OUT_OF_BOUNDS = {
    ("for (int32_t j = 0; j < t->J; ++j)", "for (int32_t j = 0; j <= t->J; ++j)"),
    ("for (int32_t k = 0; k < t->P; ++k) {", "for (int32_t k = 0; k <= t->P; ++k) {"),
    ("for (int32_t k = 0; k < P; ++k) {", "for (int32_t k = 0; k <= P; ++k) {"),
    ("for (int32_t j = 0; j < J; ++j)", "for (int32_t j = 0; j <= J; ++j)"),
    ("for (int32_t r = 0; r < R; ++r) {", "for (int32_t r = 0; r <= R; ++r) {"),
}


def survives(n, i, new_line, lines, tmp):
    mutated = lines[:i] + [new_line] + lines[i + 1:]
    c, so = os.path.join(tmp, f"m{n}.c"), os.path.join(tmp, f"m{n}.so")
    open(c, "w").write("\n".join(mutated))
    if subprocess.run(["gcc", *oracle.CFLAGS, c, "-o", so, "-lm"], capture_output=True).returncode:
        return None
    try:
        r = subprocess.run([sys.executable, "-m", "tests.oracle_mutation_sweep", "--child", so], cwd=ROOT,
                           capture_output=True, text=True, timeout=300)
    except subprocess.TimeoutExpired:
        return None
    return (lines[i].strip(), new_line.strip(), mutated) if "FAILING_PINS 0" in r.stdout else None


@pytest.fixture(scope="module")
def survivors(tmp_path_factory):
    lines = open(os.path.join(ROOT, "oracle", "esp_oracle.c")).read().split("\n")
    tmp = str(tmp_path_factory.mktemp("sweep"))
    shutil.copy(os.path.join(ROOT, "oracle", "esp_oracle.h"), tmp)
    with cf.ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        futs = [ex.submit(survives, n, i, m, lines, tmp) for n, (i, m) in enumerate(sweep.candidates(lines))]
        found = [f.result() for f in futs]
    return [s for s in found if s is not None], len(futs)


def test_every_surviving_mutant_is_known(survivors):
    found, total = survivors
    assert total >= 100
    unknown = [(a, b) for a, b, _ in found if (a, b) not in EQUIVALENT | OUT_OF_BOUNDS]
    assert not unknown, f"mutants that no pin catches: {unknown}"


def test_out_of_bounds_survivors_are_reported_by_the_sanitizers(survivors):
    rt = san._runtime("libasan.so")
    if rt is None:
        pytest.skip("gcc has no AddressSanitizer runtime")
    found, _ = survivors
    oob = [(a, b, m) for a, b, m in found if (a, b) in OUT_OF_BOUNDS]
    assert oob
    for k, (a, b, mutated) in enumerate(oob):
        d = tempfile.mkdtemp()
        c = os.path.join(d, "esp_oracle.c")
        open(c, "w").write("\n".join(mutated))
        shutil.copy(os.path.join(ROOT, "oracle", "esp_oracle.h"), d)
        so = os.path.join(d, "liboracle_san.so")
        subprocess.check_call(["gcc", *oracle.CFLAGS, *san.SAN, c, "-o", so, "-lm"])
        r = san.run_child(rt, so, os.path.join(d, "out.npz"), pins=True)
        assert r.returncode != 0 and ("AddressSanitizer" in r.stderr or "runtime error" in r.stderr), (a, b)
        shutil.rmtree(d, ignore_errors=True)
