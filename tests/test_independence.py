"""The oracle and the CUDA path share no code and neither imports the other."""
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _sources(d, exts):
    for dp, _, fs in os.walk(os.path.join(ROOT, d)):
        for f in fs:
            if f.endswith(exts):
                yield os.path.join(dp, f)


def test_product_never_imports_oracle():
    pat = re.compile(r"^\s*(import\s+oracle|from\s+oracle\b)|[\"']oracle[/\"']", re.M)
    for p in _sources("paper_2510_03275_gb300", (".py", ".cu", ".cuh", ".cpp", ".h")):
        with open(p) as f:
            assert not pat.search(f.read()), p


def test_oracle_never_imports_product():
    pat = re.compile(r"^\s*(import|from)\s+paper_2510_03275_gb300|#\s*include\s*[<\"].*sdq", re.M)
    for p in _sources("oracle", (".py", ".c", ".h")):
        with open(p) as f:
            assert not pat.search(f.read()), p
