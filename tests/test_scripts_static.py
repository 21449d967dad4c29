"""The benchmark and the build/smoke entry run only on a GPU machine; a static
check here catches a call to a helper that no longer exists before that."""
import ast
import builtins
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _undefined_calls(path):
    tree = ast.parse(open(path).read(), path)
    module = set(dir(builtins))
    for node in tree.body:
        if isinstance(node, (ast.FunctionDef, ast.AsyncFunctionDef, ast.ClassDef)):
            module.add(node.name)
        elif isinstance(node, (ast.Import, ast.ImportFrom)):
            module.update((a.asname or a.name).split(".")[0] for a in node.names)
        elif isinstance(node, (ast.Assign, ast.AnnAssign, ast.AugAssign)):
            for t in ast.walk(node):
                if isinstance(t, ast.Name) and isinstance(t.ctx, ast.Store):
                    module.add(t.id)
    missing = []
    for fn in ast.walk(tree):
        if not isinstance(fn, (ast.FunctionDef, ast.AsyncFunctionDef)):
            continue
        local = set()
        for n in ast.walk(fn):
            if isinstance(n, ast.arg):
                local.add(n.arg)
            elif isinstance(n, ast.Name) and isinstance(n.ctx, ast.Store):
                local.add(n.id)
            elif isinstance(n, (ast.FunctionDef, ast.AsyncFunctionDef, ast.ClassDef)):
                local.add(n.name)
            elif isinstance(n, (ast.Import, ast.ImportFrom)):
                local.update((a.asname or a.name).split(".")[0] for a in n.names)
        for n in ast.walk(fn):
            if isinstance(n, ast.Call) and isinstance(n.func, ast.Name):
                if n.func.id not in local and n.func.id not in module:
                    missing.append((fn.name, n.func.id, n.lineno))
    return missing


@pytest.mark.parametrize("script", ["bench.py", "__graft_entry__.py"])
def test_scripts_call_only_defined_names(script):
    assert _undefined_calls(os.path.join(ROOT, script)) == []


def test_checker_sees_a_missing_helper(tmp_path):
    p = tmp_path / "s.py"
    p.write_text("def f(x):\n    return g(x) + len(x)\n")
    assert _undefined_calls(str(p)) == [("f", "g", 2)]
