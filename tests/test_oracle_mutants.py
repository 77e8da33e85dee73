"""The oracle's pins catch plausible mistakes: every mistake planted by tests/oracle_mutants.py
(a dropped term, a wrong sign, index, bound or rounding rule, a transposed operand) makes the
pin suite fail, and the suite passes with the plugin loaded and nothing planted.  The mistakes
are planted in the oracle, on the CPU, in child processes; the oracle's files are not edited."""
import concurrent.futures
import os
import subprocess
import sys

import oracle_mutants

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TESTS = os.path.join(ROOT, "tests")
PINS = ["tests/test_oracle_formats.py", "tests/test_oracle_schedule.py", "tests/test_oracle_select.py",
        "tests/test_oracle_gemm.py"]


def run_pins(mutant):
    path = [TESTS, ROOT] + ([os.environ["PYTHONPATH"]] if os.environ.get("PYTHONPATH") else [])
    env = dict(os.environ, ORACLE_MUTANT=mutant, PYTHONPATH=os.pathsep.join(path))
    cmd = [sys.executable, "-m", "pytest", *PINS, "-x", "-q", "-p", "no:cacheprovider", "-p", "oracle_mutants"]
    return subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)


def first_failure(out):
    return next((line for line in out.splitlines() if line.startswith("FAILED")), "")


def test_pins_pass_with_nothing_planted():
    r = run_pins("none")
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]


def test_every_planted_mistake_fails_a_pin():
    workers = max(1, min(8, os.cpu_count() or 1))
    with concurrent.futures.ThreadPoolExecutor(workers) as ex:
        results = dict(zip(oracle_mutants.MUTANTS, ex.map(run_pins, oracle_mutants.MUTANTS)))
    survivors = [m for m, r in results.items() if r.returncode != 1 or not first_failure(r.stdout)]
    assert not survivors, "mistakes no pin catches: %s" % survivors
    assert len(results) >= 31
