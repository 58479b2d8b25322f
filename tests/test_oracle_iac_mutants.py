"""The IAC pins are strong enough: each plausible mistake planted in a copy of the oracle's source
(a dropped term, a wrong operand, a swapped block, ...) fails at least one check of test_oracle_iac.
The copy is built in memory from the source text; nothing of the oracle on disk changes."""

import os
import sys
import types

import pytest

from oracle import iac_oracle
from tests import test_oracle_iac as pins

SRC = os.path.join(os.path.dirname(iac_oracle.__file__), "iac_oracle.py")

MUTANTS = {
    "blocks_swapped": ("x[0:N_JOB] = a\n    x[N_JOB:2 * N_JOB] = b", "x[0:N_JOB] = b\n    x[N_JOB:2 * N_JOB] = a"),
    "mean_not_halved": ("x[k] = (a[m] + b[m]) / 2.0", "x[k] = a[m] + b[m]"),
    "framebuffer_mean": ("UTILIZATION = (SM_ACTIVE, SM_OCC, DRAM_ACTIVE, TC_ACTIVE)",
                         "UTILIZATION = (SM_ACTIVE, SM_OCC, DRAM_ACTIVE, FB_USED)"),
    "type_product": ("x[k] = a[WTYPE] + b[WTYPE]", "x[k] = a[WTYPE] * b[WTYPE]"),
    "pressure_not_divided": ("(a[FB_USED] + b[FB_USED]) / float(c_mem)", "(a[FB_USED] + b[FB_USED])"),
    "pressure_one_job": ("(a[FB_USED] + b[FB_USED]) / float(c_mem)", "a[FB_USED] / float(c_mem)"),
    "balance_inverted": ("sm_lo / sm_hi", "sm_hi / max(sm_lo, 1e-300)"),
    "balance_zero_case": ("x[k + 2] = 1.0 if sm_hi == 0.0", "x[k + 2] = 0.0 if sm_hi == 0.0"),
    "intensity_inverted": ("f[DRAM_ACTIVE] / f[SM_ACTIVE]", "f[SM_ACTIVE] / max(f[DRAM_ACTIVE], 1e-300)"),
    "intensity_no_abs": ("abs(intensity(a) - intensity(b))", "(intensity(a) - intensity(b))"),
    "intensity_zero_case": ("return 0.0 if f[SM_ACTIVE] == 0.0", "return 1.0 if f[SM_ACTIVE] == 0.0"),
    "pairwise_order": ("x[k + 2] = 1.0 if", "x[k + 3] = 1.0 if"),
    "bn_no_sqrt": ("np.sqrt(var + float(eps))", "(var + float(eps))"),
    "bn_no_eps": ("np.sqrt(var + float(eps))", "np.sqrt(var)"),
    "bn_no_beta": ("/ np.sqrt(var + float(eps)) + beta", "/ np.sqrt(var + float(eps))"),
    "bn_mean_sign": ("gamma * (z - mean)", "gamma * (z + mean)"),
    "bn_gamma_dropped": ("return gamma * (z - mean)", "return (z - mean)"),
    "hidden_relu_dropped": ("h1 = relu(batch_norm(", "h1 = (batch_norm("),
    "relu_before_bn": ("h2 = relu(batch_norm(h1 @ f64(m.W2).T + f64(m.b2), m.bn2, m.eps))",
                       "h2 = batch_norm(relu(h1 @ f64(m.W2).T + f64(m.b2)), m.bn2, m.eps)"),
    "w2_transposed": ("h1 @ f64(m.W2).T", "h1 @ f64(m.W2)"),
    "bias_dropped": ("h1 @ f64(m.W2).T + f64(m.b2)", "h1 @ f64(m.W2).T"),
    "output_without_one": ("return 1.0 + relu(h2 @ f64(m.W3) + float(m.b3))", "return relu(h2 @ f64(m.W3) + float(m.b3))"),
    "output_without_relu": ("return 1.0 + relu(h2 @ f64(m.W3) + float(m.b3))", "return 1.0 + (h2 @ f64(m.W3) + float(m.b3))"),
    "output_bias_dropped": ("h2 @ f64(m.W3) + float(m.b3)", "h2 @ f64(m.W3)"),
}


def mutant_module(name):
    old, new = MUTANTS[name]
    with open(SRC) as f:
        src = f.read()
    assert src.count(old) == 1, f"anchor of {name} not unique in the oracle"
    return module_from(src.replace(old, new), f"iac_oracle_{name}")


def module_from(src, name):
    mod = types.ModuleType(name)
    sys.modules[name] = mod          # dataclasses look their module up by name
    exec(compile(src, SRC, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_fails_a_pin(name):
    mod = mutant_module(name)
    for check in pins.CHECKS:
        try:
            check(mod)
        except Exception:
            return
    pytest.fail(f"planted mistake {name!r} passed every IAC pin")


def test_unmutated_source_passes():
    with open(SRC) as f:
        src = f.read()
    mod = module_from(src, "iac_oracle_copy")
    for check in pins.CHECKS:
        check(mod)
