"""Readers of the fixtures under tests/golden (see the citation in each file)."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                yield line.split()


def kuhn_equilibrium():
    """(value, [first-player policies], second-player policy), fp32 tables."""
    value, first, second = None, [], None
    for tok in _lines("kuhn_equilibrium.txt"):
        if tok[0] == "value":
            value = float(tok[1])
        elif tok[0] == "first":
            first.append(np.array([float(x) for x in tok[2:8]], np.float32))
        elif tok[0] == "second":
            second = np.array([float(x) for x in tok[2:8]], np.float32)
    return value, first, second


def leduc_exact_small():
    """[(seat0 id, seat1 id, exact value)] of tests/golden/leduc_exact_small.txt."""
    return [(int(t[1]), int(t[2]), float(t[3])) for t in _lines("leduc_exact_small.txt")]
