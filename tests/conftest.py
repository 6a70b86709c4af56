import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: takes more than a few seconds")


def read_golden(name, ncols=None):
    """Rows of a '|'-separated golden fixture, comments and blank lines skipped; with
    ncols, the last column keeps any further '|' characters (free-text derivation)."""
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            rows.append([c.strip() for c in line.split("|", (ncols - 1) if ncols else -1)])
    return rows


def parse_floats(s):
    return [float.fromhex(v.strip()) if "0x" in v else float(v) for v in s.split(",")]


def parse_ints(s):
    return [int(v.strip(), 0) for v in s.split(",")]
