"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake (a dropped term, a wrong sign, a wrong index, a
missing factor) into a copy of ``oracle/kdn_oracle.c`` on the CPU, rebuilds the
copy in a temporary directory and runs the pin suite against it; the suite
must fail.  Nothing here touches a GPU.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTANTS = [
    # forward: prediction, gain, innovation, read, posterior variance
    ("st->phat[i] = st->alpha[i] * st->alpha[i] * p[i] + J->omega[th * dk + i];",
     "st->phat[i] = st->alpha[i] * p[i] + J->omega[th * dk + i];"),
    ("s += st->phat[i] * kt[i] * kt[i];", "s += st->phat[i] * kt[i];"),
    ("st->delta[j] = vt[j] - acc;", "st->delta[j] = vt[j] + acc;"),
    ("o_t[j] = J->tau * acc;", "o_t[j] = acc;"),
    ("p[i] = st->phat[i] / (1.0 + st->u[i] * st->phat[i]);",
     "p[i] = st->phat[i] / (1.0 + st->u[i]);"),
    ("st->u[0] = J->mu * st->n2 / (dk * rt);", "st->u[0] = J->mu * st->n2 / rt;"),
    ("a /= dk;", "a /= 1;"),
    ("for (int i = 0; i < dk; ++i) acc += S[(size_t)i * dv + j] * qt[i];",
     "for (int i = 0; i < dk; ++i) acc += S[(size_t)i * dv + j] * kt[i];"),
    # backward
    ("dphat[i] += dkap[i] * kt[i] / st->s + ds * kt[i] * kt[i];",
     "dphat[i] += dkap[i] * kt[i] / st->s;"),
    ("dalpha[i] += 2.0 * st->alpha[i] * pprev[i] * dphat[i];",
     "dalpha[i] += st->alpha[i] * pprev[i] * dphat[i];"),
    ("dr += -dbeta * st->beta / den;", "dr += dbeta * st->beta / den;"),
    ("const double dshat = dS[(size_t)i * dv + j] - kt[i] * ddelta[j];",
     "const double dshat = dS[(size_t)i * dv + j];"),
    ("dkt[i] += du * 2.0 * J->mu * kt[i] / rt;", "dkt[i] += du * J->mu * kt[i] / rt;"),
    ("dp[i] = st->alpha[i] * st->alpha[i] * dphat[i];", "dp[i] = st->alpha[i] * dphat[i];"),
    # gradient with respect to mu
    ("J->dmu[(size_t)b * J->H + h] += du * kt[i] * kt[i] / rt;",
     "J->dmu[(size_t)b * J->H + h] += du * kt[i] / rt;"),
    ("J->dmu[(size_t)b * J->H + h] += du * st->n2 / (dk * rt);",
     "J->dmu[(size_t)b * J->H + h] += du * st->n2 / rt;"),
    # logit gates (the Python side of the oracle)
    ("__init__.py", 'out["dg"] = out["dg"] * _sigmoid(-x)', 'out["dg"] = out["dg"] * _sigmoid(x)'),
    ("__init__.py", 'out["domega"] = out["domega"] * _sigmoid(y)', 'out["domega"] = out["domega"]'),
    ("__init__.py", 'out["dr"] = out["dr"] * _sigmoid(z)', 'out["dr"] = out["dr"] * _sigmoid(-z)'),
    ("__init__.py", "return -_softplus(-x), _softplus(y), r_min + _softplus(z)",
     "return -_softplus(-x), _softplus(y), _softplus(z)"),
    ("__init__.py", "return -_softplus(-x), _softplus(y), r_min + _softplus(z)",
     "return -_softplus(x), _softplus(y), r_min + _softplus(z)"),
]


@pytest.mark.parametrize("idx", range(len(MUTANTS)))
def test_pins_catch_planted_mistake(idx, tmp_path):
    fname, src, mut = MUTANTS[idx] if len(MUTANTS[idx]) == 3 else ("kdn_oracle.c",) + MUTANTS[idx]
    (tmp_path / "oracle").mkdir()
    for f in ("kdn_oracle.c", "__init__.py"):
        text = open(os.path.join(ROOT, "oracle", f)).read()
        if f == fname:
            assert text.count(src) >= 1, "mutation site not found: " + src
            text = text.replace(src, mut, 1)
        (tmp_path / "oracle" / f).write_text(text)
    shutil.copy(os.path.join(ROOT, "kdn_inputs.py"), tmp_path)
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), tmp_path / "tests" / "golden")
    for f in ("conftest.py", "test_oracle_pins.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), tmp_path / "tests")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle_pins.py"], cwd=tmp_path, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 1, r.stdout[-2000:]
