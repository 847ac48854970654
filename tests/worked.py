"""Readers for the hand-worked fixtures under tests/golden/ (verification,
mixed sampling, token trees at V = 4).  Logits are ln(w) of small integer
weights in fp32, so every probability in a case is a ratio worked out by hand
in the fixture's header; the expected outputs come from that hand arithmetic,
not from any implementation."""
from __future__ import annotations

import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

# the weights of verify_v4_worked.txt (k = 2, V = 4)
VERIFY_DRAFT_W = [[4, 2, 1, 1], [1, 1, 1, 1]]
VERIFY_TARGET_W = [[1, 2, 3, 2], [1, 1, 2, 4], [1, 1, 1, 5]]
# mixed_v4_worked.txt
MIXED_DRAFT_W = [4, 2, 1, 1]
MIXED_TARGET_W = [1, 2, 3, 2]


def logits(weights) -> np.ndarray:
    return np.log(np.asarray(weights, dtype=np.float64)).astype(np.float32)


def _rows(path):
    with open(os.path.join(GOLDEN, path)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                yield [c.strip() for c in line.split("|")]


def _ints(s):
    return [int(x) for x in s.split()]


def _floats(s):
    return [float(x) for x in s.split()]


def verify_cases():
    """(name, T, tokens [2], uniforms [3], accepted, out_tokens [3])."""
    return [(r[0], float(r[1]), _ints(r[2]), _floats(r[3]), int(r[4]), _ints(r[5]))
            for r in _rows("verify_v4_worked.txt")]


def mixed_cases():
    """(name, T, beta, u, token)."""
    return [(r[0], float(r[1]), float(r[2]), float(r[3]), int(r[4])) for r in _rows("mixed_v4_worked.txt")]


def tree_cases():
    """(name, parent, draft weights [n, 4], target weights [n, 4], T, tokens [n]
    (node 0 = 0), uniforms [n], accepted, path [n], out_tokens [n], last_node)."""
    trees, cases = {}, []
    for r in _rows("tree_v4_worked.txt"):
        if r[0].startswith("tree "):
            name = r[0].split()[1]
            parent = _ints(r[1].replace("parent", ""))
            draft = [_ints(x) for x in r[2].replace("draft", "").split(";")]
            target = [_ints(x) for x in r[3].replace("target", "").split(";")]
            trees[name] = (parent, draft, target)
            continue
        parent, draft, target = trees[r[1]]
        cases.append((r[0], parent, draft, target, float(r[2]), [0] + _ints(r[3]), _floats(r[4]), int(r[5]),
                      _ints(r[6]), _ints(r[7]), int(r[8])))
    return cases
