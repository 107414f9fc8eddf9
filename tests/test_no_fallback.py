"""The product path has no fallback: without libpe.so the package does not import, and no
product source reaches the oracle (the oracle is test infrastructure only)."""
import os
import re
import shutil
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2609_04875_gb300")


def test_package_import_fails_without_the_library(tmp_path):
    dst = tmp_path / "paper_2609_04875_gb300"
    shutil.copytree(PKG, dst, ignore=shutil.ignore_patterns("*.so", "_build", "__pycache__"))
    env = dict(os.environ, PYTHONPATH=str(tmp_path))
    for mod in ("paper_2609_04875_gb300", "paper_2609_04875_gb300.driver"):
        r = subprocess.run([sys.executable, "-c", f"import {mod}"], capture_output=True, text=True,
                           cwd=str(tmp_path), env=env, timeout=300)
        assert r.returncode != 0, mod
        assert "is not built" in r.stderr, r.stderr[-1000:]


def test_product_sources_never_reach_the_oracle():
    pat = re.compile(r"^\s*(import\s+oracle|from\s+oracle|.*liboracle|#include\s+[\"<].*oracle)", re.M)
    hits = []
    for dirpath, _, files in os.walk(PKG):
        if "_build" in dirpath or "__pycache__" in dirpath:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                path = os.path.join(dirpath, f)
                with open(path) as fh:
                    if pat.search(fh.read()):
                        hits.append(path)
    for f in os.listdir(os.path.join(ROOT, "include")):
        with open(os.path.join(ROOT, "include", f)) as fh:
            if "oracle" in fh.read():
                hits.append(f)
    assert not hits, hits
