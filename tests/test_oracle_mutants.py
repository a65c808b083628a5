"""Planted mistakes in the oracle are caught by its pins.

Each mutant copies ``oracle/relation_oracle.c``, changes one line the way a plausible
slip would (a dropped term, a wrong sign, an off-by-one index, a transposed operand),
compiles it to a temporary library and runs every pin of ``oracle_pins`` against it.
Every planted mistake keeps all memory accesses in bounds (the mutants run in-process).
The test passes when at least one pin fails for every mutant.  CPU only.
"""
import os
import tempfile

import pytest

import oracle
from tests import oracle_pins

MUTANTS = [
    ("count index off by one",
     "const double count_shift = lambda * log((double)(r + 1));",
     "const double count_shift = lambda * log((double)(r > 0 ? r : 1));"),
    ("Self temperature dropped", "Rrow[j] = sigmoid(Urow[j] / tau_s);",
     "Rrow[j] = sigmoid(Urow[j]);"),
    ("Self uses the Exchange map", "Rrow[j] = sigmoid(Urow[j] / tau_s);",
     "Rrow[j] = silu(Urow[j]);"),
    ("count correction sign", "Rrow[j] = silu(Urow[j]) - count_shift;",
     "Rrow[j] = silu(Urow[j]) + count_shift;"),
    ("Exchange map is sigmoid", "Rrow[j] = silu(Urow[j]) - count_shift;",
     "Rrow[j] = sigmoid(Urow[j]) - count_shift;"),
    ("missing 1/sqrt(d)", "Urow[j] = dot(q + (size_t)r * d, k + (size_t)j * d, d) * inv_sqrt_d;",
     "Urow[j] = dot(q + (size_t)r * d, k + (size_t)j * d, d);"),
    ("transposed evidence U_ji",
     "Urow[j] = dot(q + (size_t)r * d, k + (size_t)j * d, d) * inv_sqrt_d;",
     "Urow[j] = dot(q + (size_t)j * d, k + (size_t)r * d, d) * inv_sqrt_d;"),
    ("SiLU derivative replaced by sigmoid derivative", "return s + x * s * (1.0 - s);",
     "return s * (1.0 - s);"),
    ("softmax gradient drops the row mean", "double dR = Fr[j] * (Hr[j] - FH);",
     "double dR = Fr[j] * Hr[j];"),
    ("dlambda sign", "dlam += -log_i * dR;", "dlam += log_i * dR;"),
    ("Self derivative drops 1/tau", "dU = dR * s * (1.0 - s) / tau_s;",
     "dU = dR * s * (1.0 - s);"),
    ("dP2 uses P2 instead of P1", "gk[(size_t)j * d + c] += dU * q[(size_t)r * d + c] * inv_sqrt_d;",
     "gk[(size_t)j * d + c] += dU * k[(size_t)r * d + c] * inv_sqrt_d;"),
    ("dI transposed", "gv[(size_t)j * d + c] += Fr[j] * G[c];",
     "gv[(size_t)r * d + c] += Fr[j] * dy[(size_t)j * d + c];"),
    ("g uses S - A", "g_i = sigmoid(a - s_i);                        /* g_i   */",
     "g_i = sigmoid(s_i - a);"),
    ("credit drops the (1-g)c term", "double dE = g[r] * p * ((1.0 - g[r]) * c_i + gdiff);",
     "double dE = g[r] * p * gdiff;"),
    ("credit Self sign", "double dU_self = -gg * c_i * S[r] * (1.0 - S[r]) / tau_s;",
     "double dU_self = gg * c_i * S[r] * (1.0 - S[r]) / tau_s;"),
    ("scan forgets to rescale z", "for (int c = 0; c < d; ++c) z[c] *= scale;", ""),
    ("scan uses the stale maximum", "double w = exp(silu(dot(qr, k + (size_t)j * d, d) * inv_sqrt_d) - mnew);",
     "double w = exp(silu(dot(qr, k + (size_t)j * d, d) * inv_sqrt_d) - m);"),
    ("factorised logZ drops the smaller term", "logz[r] = hi + log1p(exp(lo - hi));\n      }\n    }\n    if (S)",
     "logz[r] = hi;\n      }\n    }\n    if (S)"),
    ("multi-head head index mixed up",
     "int b = bh / H, h = bh % H;\n    long long off = (long long)b * sB + (long long)h * sH;\n    size_t n = (size_t)T * d;\n    double* buf = (double*)malloc(sizeof(double) * n * 4);",
     "int b = bh % B, h = bh / B;\n    long long off = (long long)b * sB + (long long)h * sH;\n    size_t n = (size_t)T * d;\n    double* buf = (double*)malloc(sizeof(double) * n * 4);"),
    ("sampled rows use the list position", "relation_row(rows[n], T, d,", "relation_row(n, T, d,"),
]


@pytest.mark.parametrize("mutant", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(mutant):
    name, old, new = mutant
    src = open(oracle.SOURCE).read()
    assert src.count(old) == 1, f"mutation site for '{name}' not unique/not found"
    with tempfile.TemporaryDirectory() as tmp:
        path = os.path.join(tmp, "mutant.c")
        with open(path, "w") as f:
            f.write(src.replace(old, new))
        lib = oracle.compile_source(path, os.path.join(tmp, "libmutant.so"))
        orc = oracle.Oracle(lib)
        caught = []
        for pin in oracle_pins.ALL_PINS:
            try:
                pin(orc)
            except (AssertionError, ValueError, FloatingPointError):
                caught.append(pin.__name__)
        assert caught, f"no pin catches the planted mistake '{name}'"
