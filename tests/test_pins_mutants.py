"""Mutation test of the oracle's pins: the oracle built with
-DORC_MUTANT=k carries one plausible mistake (below), and the pin files
(tests/test_oracle_*.py) run against that build in a subprocess must fail.
A mistake that no pin catches means the oracle is not pinned there."""
import concurrent.futures as cf
import glob
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PIN_FILES = sorted(glob.glob(os.path.join(ROOT, "tests", "test_oracle_*.py")))

MUTANTS = {
    1: "Gram off-diagonal sums with the sign of the atom product flipped",
    2: "Gram off-diagonal sums taking a wrong atom index",
    3: "b = B^T D r without the C^-1/2 normalisation",
    4: "power-of-two scale exponent one too large",
    5: "ridge eps absolute instead of relative to mean(d)",
    6: "Eq. 4 gain without the factor 2 on alpha^T b",
    7: "seed ties keep the larger selector",
    8: "records with equal gains ordered by tile descending",
    9: "progressive prefix one record longer than the budget allows",
    10: "record width rounded up one byte too far",
    11: "decoder adds half the correction",
    12: "Fisher-Yates permutation draw range one short",
    13: "Hadamard entry sign from OR instead of AND",
    14: "RTN group scale max|w| / 8 instead of / 7",
    15: "SDQ step max deviation / 128 instead of / 127",
    16: "forward substitution dropping its last term",
    17: "fixed-point grid one bit coarser",
    18: "record fields packed seed before tile",
    19: "packed GEMV subtracting the sidecar correction",
    20: "sign word bits read most-significant first",
    21: "P_F Fisher term read without the column block offset",
    22: "residual taken as W0 - W",
    23: "codes clamped to [-qmax - 1, qmax] when the exponent field clips",
    24: "U quotas shared out of B instead of B - h",
    25: "binary16 scale max|alpha| / (qmax + 1)",
    26: "SDQ mean of a short last block divided by the full block size",
    27: "fixed-point grid values truncated instead of rounded",
    28: "P_F prefixes taken out of B instead of B - h",
    29: "Eq. 4 gain with the ridge in G",
    30: "decoder normalising by 1/C instead of C^-1/2",
    31: "scale field holding e + e_bias",
    32: "decoder adding a record to the next column block",
    33: "byte budget rounded up",
    34: "SDQ step from the largest deviation above the mean only",
    35: "seed key taken from stream output s instead of s + 1",
    36: "coordinate permutation applied inverted",
    37: "Hadamard columns drawn with replacement",
    38: "candidates with a zero gain kept",
    39: "decoder dropping the last of its K records",
    40: "BF16 output truncated instead of rounded to nearest even",
    41: "U quotas rounded up",
    42: "RTN codes from the product with the rounded reciprocal of the scale",
}


def _run_pins(k):
    env = dict(os.environ, AWSRC_ORACLE_MUTANT=str(k), OMP_NUM_THREADS="1")
    return subprocess.run([sys.executable, "-m", "pytest", *PIN_FILES, "-x", "-q", "-m", "not gpu",
                           "-p", "no:cacheprovider"], env=env, cwd=ROOT, capture_output=True, text=True,
                          timeout=900)


@pytest.fixture(scope="module")
def outcomes():
    """Every mutant's pin run, the runs side by side (one OpenMP thread each)."""
    ks = sorted(MUTANTS)
    with cf.ThreadPoolExecutor(max(1, min(len(ks), os.cpu_count() or 1))) as ex:
        return dict(zip(ks, ex.map(_run_pins, ks)))


@pytest.mark.parametrize("k", sorted(MUTANTS))
def test_pins_catch_planted_mistake(outcomes, k):
    r = outcomes[k]
    assert r.returncode == 1, f"mistake {k} ({MUTANTS[k]}) not caught by any pin:\n{r.stdout[-3000:]}"
