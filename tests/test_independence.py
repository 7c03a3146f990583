"""The product path and the oracle stay apart (CPU only).

* No source of the library package (Python binding, CUDA sources) imports, includes or
  names the oracle, and the oracle names neither the package nor its CUDA sources; the
  one module both use, `synthetic`, imports neither.
* Importing the binding and loading the library leaves the oracle unloaded.
* Without the built library the binding raises instead of falling back to anything.
"""
import glob
import os
import re
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2406_14898_gb300")


def _sources(*patterns):
    out = []
    for p in patterns:
        out += glob.glob(os.path.join(ROOT, p), recursive=True)
    return sorted(f for f in out if "_build" not in f and "__pycache__" not in f)


def _code(path):
    """Source text without comments (# for Python, // and /* */ for C/CUDA) and strings
    that only document: what remains is what the file executes or includes."""
    with open(path) as fh:
        src = fh.read()
    if path.endswith(".py"):
        src = re.sub(r'"""[\s\S]*?"""', "", src)
        return "\n".join(line.split("#", 1)[0] for line in src.splitlines())
    src = re.sub(r"/\*[\s\S]*?\*/", "", src)
    return "\n".join(line.split("//", 1)[0] for line in src.splitlines())


def test_library_sources_do_not_reach_the_oracle():
    files = _sources("paper_2406_14898_gb300/*.py", "paper_2406_14898_gb300/csrc/*", "include/*.h", "bench.py")
    assert len(files) > 10
    pat = re.compile(r"^\s*(from\s+oracle\b|import\s+oracle\b)|#\s*include\s*[<\"].*oracle|flglm_oracle", re.M)
    for f in files:
        if os.path.basename(f) == "bench.py":
            continue  # bench.py's CPU legs time the oracle by design; checked below
        assert not pat.search(_code(f)), f


def test_bench_uses_the_oracle_only_in_its_cpu_legs():
    """bench.py imports the oracle only inside the class that times its CPU sample (the
    cpu_baseline leg and the reference arm), never at module level, so the GPU path of a
    run loads no oracle code unless that leg runs."""
    src = _code(os.path.join(ROOT, "bench.py"))
    imp = re.compile(r"^(\s*)(from\s+oracle\b|import\s+oracle\b)", re.M)
    found = imp.findall(src)
    assert found, "the CPU sample times the oracle"
    assert all(indent for indent, _ in found), "module-level oracle import in bench.py"
    for blk in re.split(r"\n(?=def |class )", src):
        if imp.search(blk):
            name = re.match(r"(?:def|class)\s+(\w+)", blk).group(1)
            assert re.search(r"oracle|cpu|reference|baseline", name, re.I), name


def test_oracle_does_not_reach_the_library():
    files = _sources("oracle/*.py", "oracle/*.cpp", "oracle/*.h", "synthetic/*.py")
    assert files
    pat = re.compile(r"paper_2406_14898_gb300|csrc|flglm_kernels|libflglm\.so|#\s*include\s*[<\"].*flglm\.h")
    for f in files:
        assert not pat.search(_code(f)), f
    syn = _code(os.path.join(ROOT, "synthetic", "__init__.py"))
    assert not re.search(r"^\s*(from|import)\s+(oracle|paper_2406_14898_gb300)\b", syn, re.M)


def test_binding_loads_without_the_oracle_and_fails_without_the_library():
    code = (
        "import sys\n"
        "sys.path.insert(0, sys.argv[1])\n"
        "from paper_2406_14898_gb300 import build, flglm\n"
        "build.build()\n"
        "flglm.lib()\n"
        "assert not [m for m in sys.modules if m == 'oracle' or m.startswith('oracle.')], 'oracle loaded'\n"
        "flglm._lib = None\n"
        "flglm.LIB_PATH = flglm.LIB_PATH + '.missing'\n"
        "try:\n"
        "    flglm.lib()\n"
        "except RuntimeError as e:\n"
        "    print('raised', e)\n"
        "else:\n"
        "    raise SystemExit('no error without the library')\n"
    )
    p = subprocess.run([sys.executable, "-c", code, ROOT], capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stdout + p.stderr
    assert "raised" in p.stdout and "not built" in p.stdout
