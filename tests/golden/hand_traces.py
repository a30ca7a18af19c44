"""Reader for the hand-derived trace fixtures in this folder.

Each ``hand_trace_*.txt`` holds a configuration followed by one line per step:
``step t | n | GNMR | Delta-GNMR | R | A after | C_t | A_t | Lock after``,
with exact rationals (``a/b``), ``inf``, and ``-`` for an empty set.
"""
from __future__ import annotations

import glob
import os
from dataclasses import dataclass, field
from fractions import Fraction

HERE = os.path.dirname(os.path.abspath(__file__))


def _num(tok: str):
    if tok == "inf":
        return float("inf")
    return Fraction(tok)


def _vec(field_: str):
    field_ = field_.strip()
    return [] if field_ == "-" else [_num(x) for x in field_.split()]


@dataclass
class HandStep:
    t: int
    n: list
    gnmr: list
    dgnmr: list
    risk: list
    mean_after: list
    candidates: list
    selected: list
    lock_after: list


@dataclass
class HandTrace:
    name: str
    cfg: dict = field(default_factory=dict)
    steps: list = field(default_factory=list)


def load(path: str) -> HandTrace:
    tr = HandTrace(os.path.basename(path))
    with open(path) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            if line.startswith("step"):
                parts = line.split("|")
                t = int(parts[0].split()[1])
                v = [_vec(p) for p in parts[1:]]
                tr.steps.append(HandStep(t, v[0], v[1], v[2], v[3], v[4],
                                         [int(x) for x in v[5]], [int(x) for x in v[6]],
                                         [int(x) for x in v[7]]))
            else:
                key, *vals = line.split()
                tr.cfg[key] = [_num(x) for x in vals] if key == "recoverable" else _num(vals[0])
    return tr


def all_traces():
    return [load(p) for p in sorted(glob.glob(os.path.join(HERE, "hand_trace_*.txt")))]
