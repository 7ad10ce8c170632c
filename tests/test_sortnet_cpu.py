"""The register sorting networks of the bulk append (csrc/sortnet.cuh),
compiled as host C++ and run on random and structured sets of 128 distinct
keys: the full sort and the top-64 selection must equal std::sort's order.
The networks take the smaller key of some compare-exchanges as (a + b) - max
by multiply-adds with a factor 1 given at run time; a factor of 3 must make the
check fail."""
from __future__ import annotations

import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2511_18936_gb300", "csrc")


def test_sorting_networks_match_std_sort(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    exe = str(tmp_path / "sortnet_check")
    subprocess.run([cxx, "-O1", "-std=c++17", "-I", CSRC, os.path.join(HERE, "native", "sortnet_check.cpp"),
                    "-o", exe], check=True)
    r = subprocess.run([exe, "5000", "1"], stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    assert r.returncode == 0, r.stdout
    assert r.stdout.strip() == "ok 5000"
    # the multiply-add form of the smaller key is exercised: a factor other
    # than 1 breaks the order, and the check must see it
    bad = subprocess.run([exe, "50", "3"], stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    assert bad.returncode == 1, bad.stdout
