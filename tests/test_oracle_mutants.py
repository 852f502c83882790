"""The oracle's pins must fail when a plausible mistake is planted in it.

Each case copies oracle/ember_oracle.c into a temporary directory, changes one
expression into a mistake someone could make reading Algorithm 1 of the paper
(a dropped term, a wrong divisor or power, a transposed index, eps inside the
square root, a sign flip, ...), compiles that copy, and runs
tests/test_oracle_pins.py against it in a child process.  The pins pass on the
real oracle and must fail on every mutant.  Nothing here touches a GPU.
"""
import os
import subprocess
import sys

import pytest

from oracle.build import CFLAGS, SRC

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")

MUTANTS = {
    "row mean divided by V": ("double mean_row = sum / (double)D;", "double mean_row = sum / (double)V;"),
    "column mean divided by D": ("double mean_col = colsum[j] / (double)V;", "double mean_col = colsum[j] / (double)D;"),
    "EMA weights swapped": ("beta2 * (double)r[i] + (1.0 - beta2) * mean_row",
                            "(1.0 - beta2) * (double)r[i] + beta2 * mean_row"),
    "bias correction with t-1": ("pow(beta2, (double)t)", "pow(beta2, (double)(t - 1))"),
    "bias correction with t+1": ("pow(beta2, (double)t)", "pow(beta2, (double)(t + 1))"),
    "normaliser without sqrt": ("double s = sqrt(rbar * cbar);", "double s = rbar * cbar;"),
    "normaliser dropped": ("rhat * chat / s", "rhat * chat"),
    "eps inside the sqrt": ("g / (sqrt(vtil) + eps)", "g / sqrt(vtil + eps)"),
    "sign flipped": ("maximize ? w + lr * u : w - lr * u", "maximize ? w - lr * u : w + lr * u"),
    "column factor indexed by row": ("double chat = (double)c[j] / bc;", "double chat = (double)c[i % D] / bc;"),
    "column factor not bias-corrected": ("double chat = (double)c[j] / bc;", "double chat = (double)c[j];"),
    "mean of rhat over D": ("rbar /= (double)V;", "rbar /= (double)D;"),
    "mean of r not bias-corrected": ("rbar += (double)r[i] / bc;", "rbar += (double)r[i];"),
    "|g| instead of g^2": ("sum += g * g;", "sum += fabs(g);"),
    "duplicate ids overwrite": ("Gd[id * D + j] += (double)rows[k * D + j];",
                                "Gd[id * D + j] = (double)rows[k * D + j];"),
    "bf16 ties away from zero": ("double q = rint(a / quantum);", "double q = round(a / quantum);"),
    "bf16 subnormals dropped": ("if (lead < -126)", "if (lead < -140)"),
    "LM-head gradient drops the last token": ("for (int64_t t = 0; t < T; ++t) {",
                                              "for (int64_t t = 0; t < T - 1; ++t) {"),
    "LM-head hidden state of the wrong token": ("hrow[d] = bf16_bits_to_double(hidden[t * D + d]);",
                                                "hrow[d] = bf16_bits_to_double(hidden[((t + 1) % T) * D + d]);"),
    "LM-head error of the neighbouring row": ("double delta = bf16_bits_to_double(dlogits[t * V + v]);",
                                              "double delta = bf16_bits_to_double(dlogits[t * V + (v + 1) % V]);"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    before, after = MUTANTS[name]
    with open(SRC) as f:
        src = f.read()
    assert before in src, "mutation site vanished from the oracle"
    csrc = tmp_path / "mutant.c"
    csrc.write_text(src.replace(before, after))
    lib = tmp_path / "libmutant.so"
    subprocess.run(["gcc", *CFLAGS, "-o", str(lib), str(csrc), "-lm"], check=True)
    env = dict(os.environ, EMBER_ORACLE_LIB=str(lib))
    res = subprocess.run(
        [sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", PINS],
        cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert res.returncode == 1, f"pins did not catch '{name}':\n{res.stdout[-2000:]}"
