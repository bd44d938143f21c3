"""The pins catch plausible mistakes in the oracle.

Each case plants one mistake in a copy of the oracle's C source (on the CPU,
in a temporary directory), builds that copy, and runs the pin tests against
it in a child process: at least one pin must fail. The planted text must
occur exactly once in the real source, so that a rewrite of the oracle makes
this test fail loudly instead of passing on a mutation that no longer applies.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "aladdin_oracle.c")

MUTATIONS = {
    # constraint (d): the banked slack theta T_dec l_out - t^dec with its sign flipped
    "bank_sign": ("bank = p->theta * p->T_dec * (double)cl->gen[slot] - cl->tdec[slot];",
                  "bank = cl->tdec[slot] - p->theta * p->T_dec * (double)cl->gen[slot];"),
    # the same slack without the SLO knob theta
    "bank_theta": ("bank = p->theta * p->T_dec * (double)cl->gen[slot] - cl->tdec[slot];",
                   "bank = p->T_dec * (double)cl->gen[slot] - cl->tdec[slot];"),
    # TTFT (c) without the time until the worker's next iteration boundary
    "offset_dropped": ("const double off = cl->off ? cl->off[w] : 0.0;",
                       "const double off = 0.0;"),
    # the round's prefill no longer stalls the requests already decoding
    "stall_dropped": ("cl->tdec[slot] += tau;", "(void)tau;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name, tmp_path):
    old, new = MUTATIONS[name]
    with open(SRC) as f:
        src = f.read()
    assert src.count(old) == 1, "mutation site of %s not found exactly once" % name
    mutant = tmp_path / ("oracle_%s.c" % name)
    mutant.write_text(src.replace(old, new))
    env = dict(os.environ, ALADDIN_ORACLE_SRC=str(mutant))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 1, "no pin failed with mutation %s:\n%s" % (name, r.stdout[-2000:])
    assert " failed" in r.stdout
