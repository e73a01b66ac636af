"""The C ABI as a C or C++ program uses it, on CPU: `include/whtmix.h` compiles as C11 and as
C++17 with every warning an error, both link against the built `libwhtmix.so`, and the C program
(`tests/c_abi_check.c`) gets the documented status code from every host-side argument check.  No
call in either program reaches the device."""
import os
import shutil
import subprocess

import pytest

from paper_2607_25234_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")
C_SRC = os.path.join(ROOT, "tests", "c_abi_check.c")

CXX_SRC = r"""
#include "whtmix.h"
#include <cstdio>
int main() {
  // extern "C" linkage: unmangled names resolve from C++
  size_t bytes = 0;
  if (whtmix_plan(256, 64) != 2) return 1;
  if (whtmix_workspace_bytes(1, 65536, 128, WHTMIX_BF16, 0, &bytes) != WHTMIX_OK) return 2;
  if (bytes != 256 + (size_t{1} << 23) * 4) return 3;
  std::printf("c++ abi ok\n");
  return 0;
}
"""


def link_flags():
    libdir = os.path.dirname(libbuild.LIB)
    return ["-L", libdir, "-lwhtmix", f"-Wl,-rpath,{libdir}"]


@pytest.fixture(scope="module")
def built():
    libbuild.build()


@pytest.mark.skipif(shutil.which("gcc") is None, reason="no C compiler")
def test_c_program_links_and_gets_the_documented_status_codes(built, tmp_path):
    exe = tmp_path / "c_abi_check"
    subprocess.run(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", INCLUDE, C_SRC, "-o", str(exe)]
                   + link_flags(), check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == "c abi ok"


@pytest.mark.skipif(shutil.which("g++") is None, reason="no C++ compiler")
def test_cxx_program_links_with_c_linkage(built, tmp_path):
    src = tmp_path / "abi.cpp"
    src.write_text(CXX_SRC)
    exe = tmp_path / "abi_cpp"
    subprocess.run(["g++", "-std=c++17", "-Wall", "-Wextra", "-Werror", "-I", INCLUDE, str(src), "-o", str(exe)]
                   + link_flags(), check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == "c++ abi ok"
