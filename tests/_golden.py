"""Loads the hand-computed fixtures under tests/golden/."""
import ast
import json
import math
import os
from fractions import Fraction

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def value(expr) -> float:
    """Evaluates a fixture entry: a number, a fraction "a/b", or an expression
    of fractions, + - * / and ln(...)."""
    if isinstance(expr, (int, float)):
        return float(expr)
    tree = ast.parse(expr, mode="eval")

    def ev(node):
        if isinstance(node, ast.Expression):
            return ev(node.body)
        if isinstance(node, ast.Constant):
            return Fraction(node.value)
        if isinstance(node, ast.BinOp):
            a, b = ev(node.left), ev(node.right)
            op = type(node.op)
            if op is ast.Add:
                return a + b
            if op is ast.Sub:
                return a - b
            if op is ast.Mult:
                return a * b
            if op is ast.Div:
                return a / b
        if isinstance(node, ast.UnaryOp) and isinstance(node.op, ast.USub):
            return -ev(node.operand)
        if isinstance(node, ast.Call) and getattr(node.func, "id", "") == "ln":
            return math.log(float(ev(node.args[0])))
        raise ValueError(f"unsupported fixture expression {expr!r}")
    return float(ev(tree))
