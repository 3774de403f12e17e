"""Mutation test of the oracle's pins: a copy of the oracle's source with one
plausible mistake planted in it (tests/oracle_mutants.py) is built, and the
pin files (tests/test_oracle_*.py) run against that build in a subprocess
must fail. A mistake that no pin catches means the oracle is not pinned there.
The oracle itself carries no planted mistake."""
import concurrent.futures as cf
import glob
import os
import subprocess
import sys

import pytest

from oracle_mutants import MUTANTS

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PIN_FILES = sorted(glob.glob(os.path.join(ROOT, "tests", "test_oracle_*.py")))
SRC = os.path.join(ROOT, "oracle", "awsrc_oracle.c")



def _mutant_source(k, tmpdir):
    """The oracle's source with mistake k planted: each edit replaces exactly
    one occurrence of its text."""
    s = open(SRC).read()
    for old, new in MUTANTS[k][1]:
        assert s.count(old) == 1, f"mistake {k}: its edit no longer matches the oracle's source once"
        s = s.replace(old, new)
    path = os.path.join(tmpdir, f"oracle_mutant{k}.c")
    with open(path, "w") as f:
        f.write(s)
    return path


def _run_pins(k, tmpdir):
    env = dict(os.environ, AWSRC_ORACLE_SRC=_mutant_source(k, tmpdir), OMP_NUM_THREADS="1")
    return subprocess.run([sys.executable, "-m", "pytest", *PIN_FILES, "-x", "-q", "-m", "not gpu",
                           "-p", "no:cacheprovider"], env=env, cwd=ROOT, capture_output=True, text=True,
                          timeout=900)


@pytest.fixture(scope="module")
def outcomes(tmp_path_factory):
    """Every mutant's pin run, the runs side by side (one OpenMP thread each)."""
    tmpdir = str(tmp_path_factory.mktemp("oracle_mutants"))
    ks = sorted(MUTANTS)
    with cf.ThreadPoolExecutor(max(1, min(len(ks), os.cpu_count() or 1))) as ex:
        return dict(zip(ks, ex.map(lambda k: _run_pins(k, tmpdir), ks)))


def test_oracle_source_carries_no_planted_mistake():
    s = open(SRC).read()
    assert "MUTANT" not in s
    for k, (what, edits) in MUTANTS.items():
        assert all(s.count(old) == 1 for old, _ in edits), (k, what)


@pytest.mark.parametrize("k", sorted(MUTANTS))
def test_pins_catch_planted_mistake(outcomes, k):
    r = outcomes[k]
    assert r.returncode == 1, f"mistake {k} ({MUTANTS[k][0]}) not caught by any pin:\n{r.stdout[-3000:]}"
