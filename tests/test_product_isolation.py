"""The product path does not use the oracle: nothing in the library package (its
Python modules and CUDA / C++ sources) imports, loads or names oracle/ as code."""
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2609_32479_gb300")


def _sources():
    for dirpath, _, files in os.walk(PKG):
        if "__pycache__" in dirpath or "_lib" in dirpath:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp", ".c")):
                yield os.path.join(dirpath, f)


def test_package_never_imports_the_oracle():
    pat = re.compile(r"^\s*(from\s+oracle\b|import\s+oracle\b)|trackfit_oracle|seed_oracle|#include\s+\"[^\"]*oracle",
                     re.M)
    hits = [p for p in _sources() if pat.search(open(p).read())]
    assert not hits, hits


def test_oracle_never_imports_the_package():
    pat = re.compile(r"^\s*(from|import)\s+paper_2609_32479_gb300\b", re.M)
    for f in os.listdir(os.path.join(ROOT, "oracle")):
        if f.endswith(".py"):
            assert not pat.search(open(os.path.join(ROOT, "oracle", f)).read()), f
