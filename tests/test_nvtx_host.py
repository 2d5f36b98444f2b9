"""NVTX ranges of the Python binding: off by default (the public functions are
the plain ones), on with CMC_NVTX=1 at import (each wrapped once, keeping its
name).  Checked in fresh interpreters, without calling the device."""

import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
NAMES = ["denoise", "bridge_epilogue", "score_select", "question_select", "two_tier_decode_attn",
         "decode_step", "tier1_gather", "window_append", "stage_copies"]


def _probe(env_value):
    code = ("import paper_2609_25537_gb300.cmc as c\n"
            f"names = {NAMES!r}\n"
            "print(','.join(str(hasattr(getattr(c, n), '__wrapped__')) for n in names))\n"
            "print(','.join(getattr(c, n).__name__ for n in names))\n")
    env = dict(os.environ)
    env.pop("CMC_NVTX", None)
    if env_value is not None:
        env["CMC_NVTX"] = env_value
    out = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    wrapped, names = out.stdout.strip().splitlines()
    return wrapped.split(","), names.split(",")


@pytest.mark.parametrize("value,expect", [(None, "False"), ("0", "False"), ("1", "True")])
def test_nvtx_ranges_switch(value, expect):
    wrapped, names = _probe(value)
    assert wrapped == [expect] * len(NAMES)
    assert names == NAMES
