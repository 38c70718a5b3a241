"""The C ABI's host code under AddressSanitizer and UndefinedBehaviorSanitizer.

build(variant="asan") compiles the host side of the boundary (argument and
shape checks, the thread-local error messages, workspace layouts and size
queries) with -fsanitize=address,undefined. A sanitized C program then drives
every entry point through the paths that end on the host, before any device
work: NULL, unaligned and out-of-range arguments, invalid and extreme shapes,
and the size queries over a sweep of shapes. Any sanitizer report fails the
test. No GPU is needed.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stdint.h>
#include <stdio.h>
#include <string.h>
#include "hilo.h"

static int calls = 0, errors = 0;
#define CALL(expr) do { int rc_ = (expr); ++calls; if (rc_ != HILO_OK) { ++errors; \
    if (strlen(hilo_last_error()) == 0) { printf("no message: %s\n", #expr); return 1; } } } while (0)

int main(void) {
  hilo_shape good = {2, 8, 12, 256, 4, 2, 1, 1, 0};
  hilo_shape lf = {2, 8, 12, 256, 4, 2, 1, 1, 4};
  hilo_shape bad[] = {
    {0, 8, 8, 128, 4, 1, 1, 1, 0}, {1, 7, 8, 128, 4, 1, 1, 1, 0}, {1, 8, 8, 100, 4, 1, 1, 1, 0},
    {1, 8, 8, 8192, 4, 1, 1, 1, 0}, {1, 8, 8, 128, 4, 1, 1, 3, 0}, {1, 6, 8, 128, 4, 1, 1, 2, 0},
    {1, 256, 256, 128, 4, 1, 1, 1, 0}, {1, 8, 12, 128, 4, 1, 1, 1, 3}, {1, 8, 12, 128, 4, 1, 1, 2, 4},
    {140000, 128, 128, 128, 4, 1, 1, 1, 0}, {1, 8, 8, 128, -1, 1, 1, 1, 0}, {1, 8, 8, 256, 4, 3, 1, 1, 0},
    {1, 8, 8, 128, 4, 4, 1, 1, 0}, {1, 8, 8, 128, 4, 1, 2, 1, 0}, {-5, -5, -5, -5, -5, -5, -5, -5, -5},
    {2147483647, 2147483647, 2147483646, 2147483647, 2147483647, 1, 1, 1, 0}};
  const int nbad = (int)(sizeof(bad) / sizeof(bad[0]));
  hilo_split_out sp, sp_null;
  hilo_block_weights w, w_null;
  hilo_block_weights_fp8 w8;
  void* A = (void*)(uintptr_t)4096;   /* aligned non-NULL placeholders: never dereferenced */
  void* U = (void*)(uintptr_t)4100;   /* 4-byte aligned only */
  int i, s;
  size_t total = 0;
  memset(&sp_null, 0, sizeof sp_null);
  sp.labels = (uint8_t*)A; sp.row_src = (int32_t*)A; sp.counts = (int32_t*)A; sp.cu_img = (int32_t*)A;
  sp.tok_row = (int32_t*)A;
  memset(&w_null, 0, sizeof w_null);
  memset(&w8, 0, sizeof w8);
  w = w_null;

  for (s = -9; s <= 2; ++s) total += strlen(hilo_status_string(s));
  total += strlen(hilo_last_error());
  total += hilo_row_capacity(NULL) + hilo_row_capacity(&good) + hilo_row_capacity(&lf);
  total += hilo_split_workspace_bytes(&good) + hilo_sobel_workspace_bytes(NULL) + hilo_sobel_workspace_bytes(&good);
  for (i = 0; i < nbad; ++i) {
    total += hilo_row_capacity(&bad[i]) + hilo_sobel_workspace_bytes(&bad[i]);
    total += hilo_block_workspace_bytes(&bad[i], 64) + hilo_block_fp8_workspace_bytes(&bad[i], 64);
    CALL(hilo_score(&bad[i], A, (float*)A, NULL));
    CALL(hilo_split(&bad[i], (float*)A, (uint8_t*)A, (int32_t*)A, (int32_t*)A, &sp, NULL, 0, NULL));
    CALL(hilo_split_regions(&bad[i], (float*)A, (uint8_t*)A, (int32_t*)A, (int32_t*)A, &sp, NULL, 0, NULL));
    CALL(hilo_pack(&bad[i], A, &sp, A, 64, NULL));
    CALL(hilo_block_forward(&bad[i], &w, (int32_t*)A, 64, A, A, HILO_BF16, (float*)A, A, 1u << 30, NULL));
    CALL(hilo_block_forward_fp8(&bad[i], &w8, (int32_t*)A, 64, A, A, HILO_BF16, (float*)A, A, 1u << 30, NULL));
    CALL(hilo_unpack(&bad[i], (float*)A, &sp, (float*)A, NULL));
  }
  for (i = 0; i < 64; ++i) {   /* size queries over a sweep of valid shapes and capacities */
    hilo_shape t = good;
    t.B = 1 + i % 5; t.H = 2 * (1 + i % 32); t.W = 4 * (1 + i % 16); t.d = 128 * (1 + i % 32);
    t.T = 37 * i; t.heads = t.d / 128; t.mlp = i & 1;
    total += hilo_row_capacity(&t) + hilo_block_workspace_bytes(&t, 97 * i) + hilo_block_fp8_workspace_bytes(&t, 97 * i);
    total += hilo_block_workspace_bytes(&t, -1);
  }
  CALL(hilo_score(NULL, A, (float*)A, NULL));
  CALL(hilo_score(&good, NULL, (float*)A, NULL));
  CALL(hilo_split(&good, (float*)A, (uint8_t*)A, (int32_t*)A, (int32_t*)A, NULL, NULL, 0, NULL));
  CALL(hilo_split(&good, (float*)A, (uint8_t*)A, (int32_t*)A, (int32_t*)A, &sp_null, NULL, 0, NULL));
  CALL(hilo_split_regions(&lf, (float*)A, (uint8_t*)A, (int32_t*)A, (int32_t*)A, &sp, NULL, 0, NULL));
  CALL(hilo_sobel_select(&good, (float*)A, 0, 16, (uint8_t*)A, 1, 0.1f, (uint8_t*)A, A, 1u << 20, NULL));
  CALL(hilo_sobel_select(&good, (float*)A, 3, 12, (uint8_t*)A, 1, 0.1f, (uint8_t*)A, A, 1u << 20, NULL));
  CALL(hilo_sobel_select(&good, (float*)A, 3, 16, (uint8_t*)A, 99, 0.1f, (uint8_t*)A, A, 1u << 20, NULL));
  CALL(hilo_sobel_select(&good, (float*)A, 3, 16, (uint8_t*)A, 1, 0.1f, (uint8_t*)A, U, 1u << 20, NULL));
  CALL(hilo_pack(&good, NULL, &sp, A, 64, NULL));
  CALL(hilo_block_forward(&good, &w_null, (int32_t*)A, 64, A, A, HILO_BF16, (float*)A, A, 1u << 30, NULL));
  CALL(hilo_block_forward(&good, &w, (int32_t*)A, -3, A, A, HILO_BF16, (float*)A, A, 1u << 30, NULL));
  CALL(hilo_block_forward(&good, &w, (int32_t*)A, 64, A, A, 7, (float*)A, A, 1u << 30, NULL));
  CALL(hilo_block_forward(&good, &w, (int32_t*)A, 64, U, A, HILO_BF16, (float*)A, A, 1u << 30, NULL));
  CALL(hilo_block_forward_prop(&good, &w, (int32_t*)A, 64, A, A, HILO_BF16, NULL, (float*)A, A, 1u << 30, NULL));
  CALL(hilo_block_forward_fp8(&good, &w8, (int32_t*)A, 64, A, A, HILO_BF16, (float*)A, A, 1u << 30, NULL));
  CALL(hilo_block_forward_static_ws(NULL, &w, (int32_t*)A, 64, A, A, HILO_BF16, (float*)A, NULL));
  CALL(hilo_row_sizes(&good, &sp, NULL, 64, NULL));
  CALL(hilo_row_sizes(&good, &sp, (float*)A, -1, NULL));
  CALL(hilo_unpack(&good, NULL, &sp, (float*)A, NULL));
  CALL(hilo_unpack_delta(&good, (float*)A, U, A, &sp, (float*)A, NULL));
  CALL(hilo_unpack_update(&good, NULL, &sp, A, 0.5f, NULL));
  CALL(hilo_quantize_rows_e4m3(NULL, HILO_BF16, 4, 64, (uint8_t*)A, (float*)A, NULL));
  CALL(hilo_quantize_rows_e4m3(U, HILO_BF16, 4, 64, (uint8_t*)A, (float*)A, NULL));
  CALL(hilo_quantize_rows_e4m3(A, HILO_BF16, 4, 60, (uint8_t*)A, (float*)A, NULL));
  CALL(hilo_quantize_rows_e4m3(A, 9, 4, 64, (uint8_t*)A, (float*)A, NULL));
  CALL(hilo_convert_bf16_to_f16(NULL, A, 64, NULL));
  CALL(hilo_convert_bf16_to_f16(U, A, 64, NULL));
  CALL(hilo_set_stage_events(NULL, 3));
  CALL(hilo_set_stage_events(NULL, 17));
  CALL(hilo_set_stage_events(NULL, -1));
  total += hilo_launch_count();
  printf("calls %d errors %d sizes %zu\nok\n", calls, errors, total);
  return 0;
}
"""


def test_host_code_clean_under_asan_and_ubsan(tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    probe = subprocess.run([gcc, "-fsanitize=address", "-fsanitize=undefined", "-x", "c", "-", "-o",
                            str(tmp_path / "probe")], input="int main(void){return 0;}", capture_output=True,
                           text=True)
    if probe.returncode != 0:
        pytest.skip("the C compiler has no sanitizer runtime")
    from paper_2606_13898_gb300 import build
    lib = build.build(variant="asan")
    src = tmp_path / "host.c"
    src.write_text(PROGRAM)
    exe = tmp_path / "host"
    libdir = os.path.dirname(lib)
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-fsanitize=address", "-fsanitize=undefined",
                        "-fno-omit-frame-pointer", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe),
                        "-L", libdir, "-lhilo", f"-Wl,-rpath,{libdir}"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    env = dict(os.environ, ASAN_OPTIONS="detect_leaks=0:abort_on_error=0:halt_on_error=1",
               UBSAN_OPTIONS="halt_on_error=1:print_stacktrace=1")
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300, env=env)
    report = r.stdout[-3000:] + r.stderr[-6000:]
    assert r.returncode == 0, report
    assert "AddressSanitizer" not in r.stderr and "runtime error" not in r.stderr, report
    lines = r.stdout.strip().splitlines()
    assert lines[-1] == "ok", report
    calls, errors = (int(v) for v in lines[-2].split()[1:4:2])
    assert calls >= 130 and errors == calls  # every driven call ends on the host with a status and a message
