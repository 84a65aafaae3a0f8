"""The boundary is usable from plain C: include/videomla.h compiles as C11
with every warning an error, and a C program linked against libvideomla.so
calls the host-only entry points (no GPU needed) and gets the documented
results."""

import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")
LIBDIR = os.path.join(ROOT, "paper_2605_30351_gb300")

C_SOURCE = r"""
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include "videomla.h"

static mla_config wan(void) {
  mla_config c;
  memset(&c, 0, sizeof c);
  c.hidden = 1536; c.heads = 12; c.head_dim = 128; c.d_c = 192; c.d_r = 32; c.d_q = 768;
  c.rope_pairs_t = 6; c.rope_pairs_h = 5; c.rope_pairs_w = 5;
  c.rope_dim_t = 44; c.rope_dim_h = 42; c.rope_dim_w = 42;
  c.rope_theta = 10000.0; c.rope_table_len = 1024;
  c.tokens_per_frame = 1560; c.window_frames = 21; c.batch = 1; c.rms_eps = 1e-6f;
  return c;
}

int main(void) {
  mla_config c = wan();
  if (mla_version() <= 0) return 10;
  if (mla_config_check(&c) != MLA_OK) return 11;
  unsigned long long bytes = mla_rope_table_bytes(&c);
  if (bytes != 1024ull * 16 * 2 * sizeof(float)) return 12;
  float* table = (float*)malloc(bytes);
  if (!table || mla_rope_table_fill(&c, table) != MLA_OK) return 13;
  /* position 0: every pair at angle 0 -> (cos, sin) = (1, 0) */
  for (int i = 0; i < 16; ++i)
    if (table[2 * i] != 1.0f || table[2 * i + 1] != 0.0f) return 14;
  free(table);
  mla_config bad = c;
  bad.rope_pairs_t = 7; /* 2 * (7 + 5 + 5) != d_r */
  if (mla_config_check(&bad) != MLA_ERR_ARG) return 15;
  if (mla_config_check(NULL) != MLA_ERR_ARG) return 16;
  if (mla_rope_table_bytes(&bad) != 0) return 17;
  const char* s = mla_status_string(MLA_ERR_RANGE);
  if (!s || !s[0]) return 18;
  printf("ok %d\n", mla_version());
  return 0;
}
"""


def test_header_compiles_as_c_and_links(tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    lib = os.path.join(LIBDIR, "libvideomla.so")
    if not os.path.exists(lib):
        pytest.skip("libvideomla.so is not built")
    src = tmp_path / "use_abi.c"
    src.write_text(C_SOURCE)
    exe = tmp_path / "use_abi"
    r = subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-pedantic",
                        f"-I{INCLUDE}", str(src), f"-L{LIBDIR}", "-lvideomla",
                        f"-Wl,-rpath,{LIBDIR}", "-o", str(exe)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, (r.returncode, r.stdout, r.stderr)
    assert r.stdout.startswith("ok ")
