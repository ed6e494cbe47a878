"""Parser for the hand-worked examples in tests/golden/hand_examples.txt."""

from __future__ import annotations

import math
import os
from dataclasses import dataclass

import numpy as np

GOLDEN_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@dataclass
class HandExample:
    name: str
    tokens: np.ndarray      # float64 [N, d]
    b: list
    r: list
    n_out: int
    clusters: list          # list of lists of input rows, in output order
    x_out: np.ndarray | None


def load_hand_examples(path: str | None = None) -> list:
    path = path or os.path.join(GOLDEN_DIR, "hand_examples.txt")
    examples, cur, mode = [], None, None
    with open(path) as f:
        lines = [ln.split("#", 1)[0].rstrip() for ln in f if not ln.lstrip().startswith("#")]
    lines.append("")
    for ln in lines:
        if not ln.strip():
            if cur is not None:
                examples.append(_finish(cur))
                cur, mode = None, None
            continue
        head, *rest = ln.split()
        if head == "example":
            cur = {"name": rest[0], "tokens": [], "x_out": []}
        elif head == "tokens":
            mode = "tokens"
        elif head == "x_out":
            mode = "x_out"
        elif head == "polar":
            cur["tokens"] = [[math.cos(math.radians(float(a))), math.sin(math.radians(float(a)))]
                             for a in rest]
            mode = None
        elif head in ("b", "r"):
            cur[head] = [int(v) for v in rest]
            mode = None
        elif head == "n_out":
            cur["n_out"] = int(rest[0])
            mode = None
        elif head == "clusters":
            groups = " ".join(rest).split("|")
            cur["clusters"] = [[int(v) for v in g.split()] for g in groups]
            mode = None
        elif mode in ("tokens", "x_out"):
            cur[mode].append([float(v) for v in ln.split()])
        else:
            raise ValueError(f"unparsed golden line: {ln!r}")
    return examples


def _finish(cur: dict) -> HandExample:
    x_out = np.array(cur["x_out"], dtype=np.float64) if cur["x_out"] else None
    return HandExample(cur["name"], np.array(cur["tokens"], dtype=np.float64), cur["b"], cur["r"],
                       cur["n_out"], cur["clusters"], x_out)
