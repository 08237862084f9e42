"""The oracle pins must catch plausible mistakes.

Each case copies the oracle source to a temporary directory, plants one
mistake (a dropped term, a wrong sign, an off-by-one in causality, a
transposed operand, a missing scale, a wrong tie or output order), builds it
and runs the pin suite against it: at least one pin has to fail. Nothing here
touches a GPU.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "selection term dropped from dq": ("dqh[e] += scale_sel * dsl[j] * kbar", "dqh[e] += 0.0 * dsl[j] * kbar"),
    "softmax-gradient sign": ("dsl[j] = w[j] * (dw[j] - wdw)", "dsl[j] = w[j] * (wdw - dw[j])"),
    "own chunk visible": ("const int64_t nvis = (t / S) < Nc ? (t / S) : Nc;",
                          "const int64_t nvis = (t / S + 1) < Nc ? (t / S + 1) : Nc;"),
    "mean-pool gradient not divided by S": ("const double share = dkb[(size_t)i * d + e] / (double)S;",
                                            "const double share = dkb[(size_t)i * d + e];"),
    "ties toward higher index": ("return (a->i < b->i) ? -1 : (a->i > b->i) ? 1 : 0;",
                                 "return (a->i > b->i) ? -1 : (a->i < b->i) ? 1 : 0;"),
    "dV without chunk weight": ("dV[row + e] += w[j] * Pj[s] * dOh[e];", "dV[row + e] += Pj[s] * dOh[e];"),
    "inner gradient without chunk weight": ("const double da = Pj[s] * (dP - w[j] * Dhj);",
                                            "const double da = Pj[s] * (dP - Dhj);"),
    "dK with dO instead of q": ("dK[row + e] += scale_attn * da * qh[e];", "dK[row + e] += scale_attn * da * dOh[e];"),
    "attention scale missing": ("P[s] = scale_attn * a;", "P[s] = a;"),
    "uniform chunk weights": ("w[j] = j < keff ? exp(s[j] - m) / z : 0.0;", "w[j] = j < keff ? 1.0 / keff : 0.0;"),
    "group query uses one head": ("for (int hh = 0; hh < G; ++hh) acc += q_row[(int64_t)(g * G + hh) * d + e];",
                                  "for (int hh = 0; hh < 1; ++hh) acc += q_row[(int64_t)(g * G + hh) * d + e];"),
    "chunk-summary gradient without q": ("dkb[(size_t)i * d + e] += scale_sel * dsl[j] * qhat[e];",
                                         "dkb[(size_t)i * d + e] += scale_sel * dsl[j];"),
    "off-by-one term dropped": ("if (softmax1) z += exp(-m);", "if (softmax1) z += 0.0;"),
    "stick-breaking remainder not shrunk": ("rest *= 1.0 - beta;", "rest *= 1.0;"),
    "stick-breaking gradient without later slots": ("dsl[j] = (1.0 - beta) * w[j] * dw[j] - beta * later;",
                                                     "dsl[j] = (1.0 - beta) * w[j] * dw[j];"),
    "stick-breaking gradient over earlier slots": ("for (int j = keff - 1; j >= 0; --j) {",
                                                   "for (int j = 0; j < keff; ++j) {"),
    "selection-chain pool share not divided by S": (
        "dK[at4(b, (int64_t)i * S + s, g, e, L, Hkv, d)] = dkbar[at4(b, i, g, e, Nc, Hkv, d)] / (double)S;",
        "dK[at4(b, (int64_t)i * S + s, g, e, L, Hkv, d)] = dkbar[at4(b, i, g, e, Nc, Hkv, d)];"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    old, new = MUTATIONS[name]
    src = open(os.path.join(ROOT, "oracle", "hsa_oracle.c")).read()
    assert src.count(old) == 1, name
    for sub in ("oracle", "synth", "tests"):
        shutil.copytree(os.path.join(ROOT, sub), tmp_path / sub,
                        ignore=shutil.ignore_patterns("_build", "__pycache__", "test_oracle_mutations.py"))
    (tmp_path / "oracle" / "hsa_oracle.c").write_text(src.replace(old, new))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-p", "no:cacheprovider", "-x",
                        "tests/test_oracle_pins.py"], cwd=tmp_path, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"no pin caught: {name}\n{r.stdout[-2000:]}"
    assert "failed" in r.stdout
