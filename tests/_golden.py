"""Reader for the hand-worked fixtures under tests/golden/.

Values are stored as small exact expressions ("290/9", "log(14)", "sqrt(2)")
so that each fixture can be checked by hand against its derivation text.
"""
import ast
import json
import math
import os
from fractions import Fraction

import numpy as np

_FUNCS = {"log": math.log, "sqrt": math.sqrt, "exp": math.exp}


def _eval(node):
    if isinstance(node, ast.Expression):
        return _eval(node.body)
    if isinstance(node, ast.Constant) and isinstance(node.value, (int, float)):
        return Fraction(node.value) if isinstance(node.value, int) else node.value
    if isinstance(node, ast.BinOp):
        a, b = _eval(node.left), _eval(node.right)
        if isinstance(node.op, ast.Add):
            return a + b
        if isinstance(node.op, ast.Sub):
            return a - b
        if isinstance(node.op, ast.Mult):
            return a * b
        if isinstance(node.op, ast.Div):
            if isinstance(a, Fraction) and isinstance(b, Fraction):
                return a / b
            return float(a) / float(b)
    if isinstance(node, ast.UnaryOp) and isinstance(node.op, ast.USub):
        return -_eval(node.operand)
    if isinstance(node, ast.Call) and isinstance(node.func, ast.Name) and node.func.id in _FUNCS:
        return _FUNCS[node.func.id](*[float(_eval(a)) for a in node.args])
    raise ValueError(f"unsupported expression: {ast.dump(node)}")


def value(expr) -> float:
    if isinstance(expr, (int, float)):
        return float(expr)
    return float(_eval(ast.parse(expr, mode="eval")))


def array(nested) -> np.ndarray:
    if isinstance(nested, list):
        return np.array([array(x) for x in nested], dtype=np.float64)
    return np.float64(value(nested))


def load(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)
