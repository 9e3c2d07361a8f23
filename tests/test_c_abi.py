"""The boundary is a C ABI: a C99 program compiles against include/bergson.h
with warnings as errors, links against the library and calls its host-only
entry points (no GPU needed)."""
import os
import shutil
import subprocess

import pytest

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

C_PROGRAM = r"""
#include <stdint.h>
#include <stdio.h>
#include <string.h>
#include "bergson.h"

int main(void) {
  size_t ws = 0;
  uint64_t s_in = 0, s_out = 0;
  bergson_layer L;
  memset(&L, 0, sizeof L);
  L.A = (const void*)(uintptr_t)0x7F0000000000ull;   /* aligned, never dereferenced */
  L.G = (const void*)(uintptr_t)0x7F0000001000ull;
  L.d_in = 768; L.d_out = 3072; L.k_in = 16; L.k_out = 16;
  L.proj_kind = BERGSON_PROJ_RADEMACHER;
  printf("version %d\n", bergson_version());
  {
    const int st = bergson_project_grads_workspace(&L, 1, 32, 2048, &ws);
    printf("project_ws %d %zu\n", st, ws);
  }
  L.proj_kind = 7;
  {
    const int st = bergson_project_grads_workspace(&L, 1, 32, 2048, &ws);
    printf("bad_kind %d %d\n", st, (int)(strlen(bergson_last_error()) > 0));
  }
  printf("score_ws %d\n", bergson_score_topk_workspace(1000, 64, 4, 5, &ws));
  printf("score_ws_k_gt_n %d\n", bergson_score_topk_workspace(4, 64, 4, 5, &ws));
  bergson_module_seeds(0, 3, &s_in, &s_out);
  printf("seeds %llu %llu\n", (unsigned long long)s_in, (unsigned long long)s_out);
  {
    int64_t plan[12 * 4];
    int n = 0;
    const int st = bergson_debug_score_plan(4000000, 8192, 1024, 100, 152, plan, 4, &n);
    printf("score_plan %d %d %lld %lld\n", st, n, (long long)plan[2], (long long)plan[6]);
  }
  return 0;
}
"""


@pytest.mark.skipif(shutil.which("gcc") is None, reason="no C compiler")
def test_c_program_uses_the_abi(tmp_path):
    src = tmp_path / "abi.c"
    exe = tmp_path / "abi"
    src.write_text(C_PROGRAM)
    lib_dir = os.path.dirname(bg.LIB_PATH)
    cc = subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic",
                         "-I" + os.path.join(ROOT, "include"), str(src), "-o", str(exe),
                         "-L" + lib_dir, "-lbergson", "-Wl,-rpath," + lib_dir],
                        capture_output=True, text=True)
    assert cc.returncode == 0, cc.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120,
                         env=dict(os.environ, CUDA_VISIBLE_DEVICES=""))
    assert run.returncode == 0, run.stderr
    out = dict(line.split(" ", 1) for line in run.stdout.splitlines())
    assert int(out["version"]) == bg.bergson_version()
    st, ws = out["project_ws"].split()
    assert int(st) == bg.BERGSON_OK and int(ws) > 0
    assert out["bad_kind"].split() == [str(bg.BERGSON_EINVAL), "1"]
    assert int(out["score_ws"]) == bg.BERGSON_OK
    assert int(out["score_ws_k_gt_n"]) == bg.BERGSON_EINVAL
    assert tuple(int(v) for v in out["seeds"].split()) == orc.module_seeds(0, 3)
    st, n, rows, grid = (int(v) for v in out["score_plan"].split())
    assert st == bg.BERGSON_OK and n == 2 and rows == 9728 and grid == 152
