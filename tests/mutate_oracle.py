"""Mutation check of the oracle's pins (not collected by pytest; run by hand):

    python tests/mutate_oracle.py [--source FILE] [--funcs F1,F2] [pytest args,
                                   default tests/test_oracle_pins.py]

(--source picks another host-side file to mutate, e.g.
paper_2606_03075_gb300/shard.py with tests/test_shard.py; --funcs keeps only
the sites inside the named functions, e.g. bench.py's roofline arithmetic.)

Plants one plausible mistake at a time in a copy of oracle/tgvkv_oracle.py
(an operator or comparison swapped, a constant, index, slice bound or axis off
by one, a term or a transpose dropped, sum/mean or max/min exchanged, and/or
exchanged, the first two arguments of a call swapped) and runs the CPU pins
against the copy.  Prints every mutant that no pin kills, with its function,
line and kind; each one must be an equivalent mutant (the same results on
every input) or a gap to close with a new pin.  Takes about ten minutes.
"""
import ast
import copy
import os
import shutil
import subprocess
import sys
import tempfile
import time

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = "oracle/tgvkv_oracle.py"

SWAP_BIN = {ast.Add: ast.Sub, ast.Sub: ast.Add, ast.Mult: ast.Div, ast.Div: ast.Mult,
            ast.FloorDiv: ast.Div}
SWAP_CMP = {ast.Lt: ast.LtE, ast.LtE: ast.Lt, ast.Gt: ast.GtE, ast.GtE: ast.Gt,
            ast.Eq: ast.NotEq, ast.NotEq: ast.Eq}
SWAP_METH = {"sum": "mean", "mean": "sum", "max": "min", "min": "max", "argmax": "argmin",
             "argmin": "argmax", "floor": "ceil", "ceil": "floor"}


class Sites(ast.NodeVisitor):
    """Every mutable site, in a fixed walk order: (node, kind, enclosing function)."""

    def __init__(self):
        self.sites, self.func = [], None

    def add(self, node, kind):
        self.sites.append((node, kind, self.func))

    def visit_FunctionDef(self, node):
        prev, self.func = self.func, node.name
        self.generic_visit(node)
        self.func = prev

    def visit_BinOp(self, node):
        if type(node.op) in SWAP_BIN:
            self.add(node, "binop")
        self.add(node, "keep_left")
        self.add(node, "keep_right")
        self.generic_visit(node)

    def visit_Compare(self, node):
        if len(node.ops) == 1 and type(node.ops[0]) in SWAP_CMP:
            self.add(node, "cmp")
        self.generic_visit(node)

    def visit_Constant(self, node):
        if isinstance(node.value, (int, float)) and not isinstance(node.value, bool):
            self.add(node, "const")

    def visit_Subscript(self, node):
        if isinstance(node.slice, (ast.Name, ast.BinOp)):
            self.add(node, "index")
        self.generic_visit(node)

    def visit_UnaryOp(self, node):
        if isinstance(node.op, ast.USub):
            self.add(node, "drop_minus")
        self.generic_visit(node)

    def visit_Attribute(self, node):
        if node.attr == "T":
            self.add(node, "drop_T")
        if node.attr in SWAP_METH:
            self.add(node, "method")
        self.generic_visit(node)

    def visit_Slice(self, node):
        if node.lower is not None:
            self.add(node, "slice_lower")
        if node.upper is not None:
            self.add(node, "slice_upper")
        self.generic_visit(node)

    def visit_BoolOp(self, node):
        self.add(node, "and_or")
        self.generic_visit(node)

    def visit_Call(self, node):
        if len(node.args) >= 2 and not node.keywords:
            self.add(node, "swap_args")
        self.generic_visit(node)

    def visit_keyword(self, node):
        if node.arg == "axis" and isinstance(node.value, ast.Constant) and \
                isinstance(node.value.value, int):
            self.add(node, "axis")
        if node.arg == "keepdims":
            self.add(node, "keepdims")
        self.generic_visit(node)


def _plus_one(expr):
    return ast.BinOp(left=expr, op=ast.Add(), right=ast.Constant(1))


class Replace(ast.NodeTransformer):
    """Replace one node (found by identity) with fn(node)."""

    def __init__(self, target, fn):
        self.target, self.fn = target, fn

    def visit(self, node):
        if node is self.target:
            return self.fn(node)
        return super().visit(node)


def mutate(tree, node, kind):
    """Apply one mutation in place (or through Replace); returns (tree, text)."""
    if kind == "binop":
        old = type(node.op)
        node.op = SWAP_BIN[old]()
        return tree, f"{old.__name__} -> {type(node.op).__name__}"
    if kind == "keep_left":
        return Replace(node, lambda n: n.left).visit(tree), "right operand dropped"
    if kind == "keep_right":
        return Replace(node, lambda n: n.right).visit(tree), "left operand dropped"
    if kind == "cmp":
        old = type(node.ops[0])
        node.ops[0] = SWAP_CMP[old]()
        return tree, f"{old.__name__} -> {type(node.ops[0]).__name__}"
    if kind == "const":
        v = node.value
        node.value = v + 1 if isinstance(v, int) else (v * 1.5 if v != 0 else 1.0)
        return tree, f"{v!r} -> {node.value!r}"
    if kind == "index":
        node.slice = _plus_one(node.slice)
        return tree, "index + 1"
    if kind == "drop_minus":
        return Replace(node, lambda n: n.operand).visit(tree), "unary minus dropped"
    if kind == "drop_T":
        return Replace(node, lambda n: n.value).visit(tree), ".T dropped"
    if kind == "method":
        old = node.attr
        node.attr = SWAP_METH[old]
        return tree, f".{old} -> .{node.attr}"
    if kind == "slice_lower":
        node.lower = _plus_one(node.lower)
        return tree, "slice lower bound + 1"
    if kind == "slice_upper":
        node.upper = _plus_one(node.upper)
        return tree, "slice upper bound + 1"
    if kind == "and_or":
        old = type(node.op)
        node.op = ast.Or() if old is ast.And else ast.And()
        return tree, f"{old.__name__} -> {type(node.op).__name__}"
    if kind == "swap_args":
        node.args[0], node.args[1] = node.args[1], node.args[0]
        return tree, "first two arguments swapped"
    if kind == "axis":
        node.value = ast.Constant(node.value.value + 1)
        return tree, "axis + 1"
    if kind == "keepdims":
        node.value = ast.Constant(False)
        return tree, "keepdims=False"
    raise ValueError(kind)


def main(pytest_args, src=SRC, funcs=None):
    work = tempfile.mkdtemp(prefix="tgvkv_mut_")
    try:
        for d in ("tests", "oracle", "paper_2606_03075_gb300", "profiles"):
            shutil.copytree(os.path.join(REPO, d), os.path.join(work, d),
                            ignore=shutil.ignore_patterns("__pycache__", "_build*"))
        for f in ("pytest.ini", "bench.py"):
            shutil.copy(os.path.join(REPO, f), work)
        base = ast.parse(open(os.path.join(REPO, src)).read())
        finder = Sites()
        finder.visit(base)
        chosen = [i for i, (_, _, f) in enumerate(finder.sites) if funcs is None or f in funcs]
        n = len(chosen)
        print(f"{n} mutants", flush=True)
        survived, killed, t0 = 0, 0, time.time()
        for i in chosen:
            tree = copy.deepcopy(base)
            walk = Sites()
            walk.visit(tree)
            node, kind, func = walk.sites[i]
            line = node.lineno
            tree, what = mutate(tree, node, kind)
            ast.fix_missing_locations(tree)
            with open(os.path.join(work, src), "w") as f:
                f.write(ast.unparse(tree))
            r = subprocess.run([sys.executable, "-m", "pytest", *pytest_args, "-x", "-q",
                                "-p", "no:cacheprovider", "-m", "not gpu"],
                               cwd=work, capture_output=True, text=True, timeout=600)
            if r.returncode == 0:
                survived += 1
                print(f"survived: {func or '<module>'} line {line}: {what}", flush=True)
            else:
                killed += 1
        print(f"killed {killed} of {n}, survived {survived}, {time.time() - t0:.0f} s")
    finally:
        shutil.rmtree(work, ignore_errors=True)


if __name__ == "__main__":
    args = sys.argv[1:]
    source, only = SRC, None
    while args[:1] in (["--source"], ["--funcs"]):
        if args[0] == "--source":
            source = args[1]
        else:
            only = set(args[1].split(","))
        args = args[2:]
    main(args or ["tests/test_oracle_pins.py"], source, only)
