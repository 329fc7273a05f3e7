"""Code boundaries: the library package never reaches the oracle (no import, no path to it),
and the oracle never imports the library; only tests, smoke() and the bench's CPU legs may use
the oracle."""
import ast
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def imported_modules(path):
    tree = ast.parse(open(path).read())
    out = set()
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            out.update(a.name.split(".")[0] for a in node.names)
        elif isinstance(node, ast.ImportFrom) and node.module and node.level == 0:
            out.add(node.module.split(".")[0])
    return out


def py_files(d):
    for base, _, files in os.walk(os.path.join(ROOT, d)):
        for f in files:
            if f.endswith(".py"):
                yield os.path.join(base, f)


def test_library_does_not_import_the_oracle():
    for f in py_files("paper_2601_03700_gb300"):
        assert "oracle" not in imported_modules(f), f
        assert "oracle/" not in open(f).read(), f


def test_oracle_does_not_import_the_library():
    for f in py_files("oracle"):
        mods = imported_modules(f)
        assert "paper_2601_03700_gb300" not in mods and "bench" not in mods, f


def test_library_imports_with_the_oracle_unavailable():
    code = ("import sys; sys.modules['oracle'] = None; import paper_2601_03700_gb300 as a; "
            "print(len(a.ABI_SYMBOLS))")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]


def test_missing_library_fails_loudly():
    """No CPU fallback: loading a library that is not built raises."""
    code = ("import paper_2601_03700_gb300 as a\n"
            "try:\n"
            "    a.load_library('/nonexistent/libadept.so')\n"
            "except RuntimeError as e:\n"
            "    print('raised', 'not built' in str(e))\n")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and "raised True" in r.stdout, (r.stdout, r.stderr[-2000:])
