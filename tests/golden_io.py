"""Parser for the hand-worked examples in tests/golden/hand_examples.txt."""

from __future__ import annotations

import ast
import math
import os
from dataclasses import dataclass

import numpy as np

GOLDEN_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

# Names a value in the golden file may use: cosd(a) is the cosine of a
# degrees, sqrt the square root; inf and nan are the IEEE specials.
_FUNCS = {"cosd": lambda a: math.cos(math.radians(a)), "sqrt": math.sqrt}
_NAMES = {"inf": math.inf, "nan": math.nan}
_BINOPS = {ast.Add: lambda a, b: a + b, ast.Sub: lambda a, b: a - b,
           ast.Mult: lambda a, b: a * b, ast.Div: lambda a, b: a / b}


def _eval(node):
    if isinstance(node, ast.Expression):
        return _eval(node.body)
    if isinstance(node, ast.Constant) and isinstance(node.value, (int, float)):
        return float(node.value)
    if isinstance(node, ast.Name) and node.id in _NAMES:
        return _NAMES[node.id]
    if isinstance(node, ast.UnaryOp) and isinstance(node.op, (ast.USub, ast.UAdd)):
        v = _eval(node.operand)
        return -v if isinstance(node.op, ast.USub) else v
    if isinstance(node, ast.BinOp) and type(node.op) in _BINOPS:
        return _BINOPS[type(node.op)](_eval(node.left), _eval(node.right))
    if (isinstance(node, ast.Call) and isinstance(node.func, ast.Name) and node.func.id in _FUNCS
            and len(node.args) == 1 and not node.keywords):
        return _FUNCS[node.func.id](_eval(node.args[0]))
    raise ValueError(f"unsupported golden value: {ast.dump(node)}")


def golden_value(text: str) -> float:
    """A number, inf/nan, or arithmetic over cosd(...) / sqrt(...), e.g. 'sqrt(2)/2'."""
    return _eval(ast.parse(text, mode="eval"))


@dataclass
class HandExample:
    name: str
    tokens: np.ndarray      # float64 [N, d]
    b: list
    r: list
    n_out: int
    clusters: list          # list of lists of input rows, in output order
    x_out: np.ndarray | None
    top1: np.ndarray | None = None      # best cosine of each row over j != i
    top2: np.ndarray | None = None      # second-best cosine (ties with the best count)
    near_tie: list | None = None        # 1 where top1 - top2 does not exceed 1e-4


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
        elif head in ("b", "r", "near_tie"):
            cur[head] = [int(v) for v in rest]
            mode = None
        elif head in ("top1", "top2"):
            cur[head] = np.array([golden_value(v) for v in rest], dtype=np.float64)
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
                       cur["n_out"], cur["clusters"], x_out, cur.get("top1"), cur.get("top2"),
                       cur.get("near_tie"))
