"""The C ABI from plain C: tests/c_client/relation_client.c is compiled with gcc against
include/relation.h only, linked to the library, and run (host-only calls; no GPU)."""
import os
import subprocess

from paper_2608_20172_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_c_client(tmp_path):
    lib = libbuild.build()
    exe = tmp_path / "relation_client"
    subprocess.run(["gcc", "-std=c11", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "c_client", "relation_client.c"), "-o", str(exe),
                    lib, "-Wl,-rpath," + os.path.dirname(lib)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, f"check {r.returncode} failed: {r.stdout}{r.stderr}"
    assert "all checks passed" in r.stdout
