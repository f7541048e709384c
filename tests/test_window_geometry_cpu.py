"""Windowed 3D attention's geometry, on the CPU: the kernel's own header
(csrc/window_tiles.cuh) compiled as plain C++ and checked against brute force.

window_geometry_check.cpp walks every unit, brick row and key box of many
grids, windows, border rules and tile shapes, and checks that each in-grid
query's window lies inside its unit's key boxes and that window_mask (driven
as the kernel drives it) sets exactly the bits of the keys inside the window.
The GPU parity tests compare the kernel's outputs with the oracle on fewer
grids; this check covers the mask arithmetic for every tile shape the host
may choose.
"""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


def test_window_masks_and_coverage(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no C++ compiler")
    exe = str(tmp_path / "window_geometry_check")
    build = subprocess.run([cxx, "-O2", "-std=c++17", "-o", exe, os.path.join(HERE, "window_geometry_check.cpp")],
                           capture_output=True, text=True)
    assert build.returncode == 0, build.stderr
    run = subprocess.run([exe], capture_output=True, text=True, timeout=600)
    assert run.returncode == 0 and run.stdout.startswith("ok"), run.stdout + run.stderr
