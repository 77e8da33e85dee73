"""Structure checks of the repository (host only): the oracle and the CUDA path share no code, the
product never routes through the oracle, and the binding fails loudly without its library.

Allowed users of `oracle/`: the tests, `__graft_entry__.smoke()` and the benchmark's CPU baseline
(`bench.oracle_sample`).  `oracle/` itself imports only numpy, scipy and its own modules."""
import ast
import os
import re
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2609_33496_gb300")


def py_files(d):
    for dirpath, dirnames, files in os.walk(d):
        dirnames[:] = [x for x in dirnames if x not in ("__pycache__", "_build")]
        for f in files:
            if f.endswith(".py"):
                yield os.path.join(dirpath, f)


def imports(path):
    """(module name, enclosing top-level function or None) for every import in the file."""
    tree = ast.parse(open(path).read(), path)
    out = []

    def visit(node, func):
        for child in ast.iter_child_nodes(node):
            f = func
            if isinstance(child, (ast.FunctionDef, ast.AsyncFunctionDef)) and func is None:
                f = child.name
            if isinstance(child, ast.Import):
                out.extend((a.name, f) for a in child.names)
            elif isinstance(child, ast.ImportFrom):
                out.append((("." * child.level) + (child.module or ""), f))
            visit(child, f)

    visit(tree, None)
    return out


def top(name):
    return name.lstrip(".").split(".")[0] if not name.startswith(".") else "."


def test_package_never_imports_the_oracle():
    for path in py_files(PKG):
        for name, _ in imports(path):
            assert top(name) != "oracle", "%s imports %s" % (os.path.relpath(path, ROOT), name)


def test_oracle_imports_only_numpy_scipy_and_itself():
    for path in py_files(os.path.join(ROOT, "oracle")):
        for name, _ in imports(path):
            assert top(name) in ("numpy", "scipy", "math", "."), \
                "%s imports %s" % (os.path.relpath(path, ROOT), name)


def test_oracle_and_csrc_share_no_files():
    """The CUDA sources include only their own headers, the ABI header and CUDA's."""
    csrc = os.path.join(PKG, "csrc")
    own = set(os.listdir(csrc)) | {"chameleon.h"}
    for f in os.listdir(csrc):
        for line in open(os.path.join(csrc, f), errors="replace"):
            s = line.strip()
            if s.startswith("#include \""):
                inc = os.path.basename(s.split('"')[1])
                assert inc in own, "%s includes %s" % (f, inc)


@pytest.mark.parametrize("script,allowed", [("bench.py", {"oracle_sample"}),
                                            ("__graft_entry__.py", {"smoke", "_smoke_checks"})])
def test_entry_scripts_use_the_oracle_only_where_allowed(script, allowed):
    for name, func in imports(os.path.join(ROOT, script)):
        if top(name) == "oracle":
            assert func is not None and func in allowed, "%s imports %s in %s" % (script, name, func)


SCRATCH = re.compile(r"(^|[^A-Za-z0-9_])_work([/\\'\"]|$)", re.M)


def test_nothing_committed_reads_the_scratch_folder():
    files = [p for d in (PKG, os.path.join(ROOT, "oracle"), os.path.join(ROOT, "tests")) for p in py_files(d)]
    files += [os.path.join(ROOT, s) for s in ("bench.py", "__graft_entry__.py")]
    for path in files:
        if os.path.abspath(path) == os.path.abspath(__file__):
            continue
        assert not SCRATCH.search(open(path).read()), path


def test_binding_raises_without_the_library(tmp_path):
    """The product path has no fallback: with the library absent the first call raises."""
    code = ("import sys; sys.path.insert(0, %r)\n"
            "import paper_2609_33496_gb300._binding as b\n"
            "b.LIB_PATH = %r\n"
            "try:\n    b.lib()\nexcept RuntimeError as e:\n    print('raised', 'no fallback' in str(e))\n"
            "else:\n    print('loaded')\n") % (ROOT, str(tmp_path / "absent.so"))
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=120)
    assert r.stdout.strip() == "raised True", r.stdout + r.stderr
