"""The boundary from C: include/hilo.h compiles as strict C99, a C program
links against libhilo.so, resolves every declared entry point and makes the
host-only calls (status strings, capacity and workspace queries, argument
errors returned before any launch). No GPU is needed."""
import os
import shutil
import subprocess

import pytest

from tests.test_abi_cpu import declared_functions

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "hilo.h"

typedef void (*fn_t)(void);

int main(void) {
  /* every declared entry point, so that the link must resolve all of them */
  fn_t all[] = { %(FNS)s };
  hilo_shape s;
  hilo_shape bad;
  int n_null = 0;
  size_t i;
  for (i = 0; i < sizeof(all) / sizeof(all[0]); ++i) n_null += all[i] == NULL;
  memset(&s, 0, sizeof s);
  s.B = 2; s.H = 8; s.W = 12; s.d = 128; s.T = 4; s.heads = 1; s.mlp = 1; s.levels = 1; s.lf = 4;
  bad = s;
  bad.H = 7;
  printf("entries %%d null %%d\n", (int)(sizeof(all) / sizeof(all[0])), n_null);
  printf("status %%s %%s %%s\n", hilo_status_string(HILO_OK), hilo_status_string(HILO_ERR_TIMEOUT),
         hilo_status_string(HILO_ERR_CHECK));
  printf("capacity %%zu %%zu\n", hilo_row_capacity(&s), hilo_row_capacity(&bad));
  printf("score_null %%d\n", hilo_score(&s, NULL, NULL, NULL));
  printf("score_shape %%d\n", hilo_score(&bad, (const void*)256, (float*)256, NULL));
  printf("error %%s\n", hilo_last_error()[0] ? "set" : "empty");
  return 0;
}
"""


def test_header_is_c99_and_links_from_c(tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    from paper_2606_13898_gb300 import build
    lib = build.build()
    names = declared_functions()
    src = tmp_path / "abi.c"
    src.write_text(PROGRAM % {"FNS": ", ".join(f"(fn_t){n}" for n in names)})
    exe = tmp_path / "abi"
    libdir = os.path.dirname(lib)
    cmd = [gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", os.path.join(ROOT, "include"),
           str(src), "-o", str(exe), "-L", libdir, "-lhilo", f"-Wl,-rpath,{libdir}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    out = dict(line.split(" ", 1) for line in r.stdout.strip().splitlines())
    assert out["entries"] == f"{len(names)} null 0"
    assert out["status"] == "HILO_OK HILO_ERR_TIMEOUT HILO_ERR_CHECK"
    assert out["capacity"] == f"{2 * (96 + 96 // 16)} 0"
    assert out["score_null"] == "-1"  # HILO_ERR_ARG
    assert out["score_shape"] == "-2"  # HILO_ERR_SHAPE
    assert out["error"] == "set"
