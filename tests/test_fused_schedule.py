"""The fused kernels' static tile schedule (FusedSched in csrc/internal.cuh),
compiled for the host from the same header: every gate-up and down tile has
exactly one worker, each worker runs its gate-up tiles before its down tiles
and both in increasing order (the order the kernels' progress argument needs:
a down tile waits only for gate-up tiles), and the workers' shares of the
work (a gate-up tile worth w down tiles) are even."""
import os
import shutil
import subprocess

import pytest

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2608_23805_gb300", "csrc")

PROGRAM = r'''
#include <cstdio>
#include <vector>
#include "internal.cuh"

// returns 0 when every property holds for (U, D, P, w)
static int check(int U, int D, int P, int w) {
  std::vector<int> seen(U + D, 0);
  long long max_load = 0, total = (long long)U * w + D;
  for (int c = 0; c < P; ++c) {
    msi::FusedSched sc(U, D, P, c, w);
    int prev = -1, steps = 0;
    bool in_down = false;
    long long load = 0;
    for (int t = sc.first(); t >= 0; t = sc.next(t)) {
      if (t <= prev || t >= U + D) return 1;        // increasing, in range
      if (t < U && in_down) return 2;               // gate-up after a down tile
      in_down = in_down || t >= U;
      seen[t] += 1;
      load += t < U ? w : 1;
      prev = t;
      if (++steps > U + D) return 3;                // no cycle
    }
    if (load > max_load) max_load = load;
  }
  for (int v : seen)
    if (v != 1) return 4;                           // every tile exactly once
  // even shares: within one down tile of the ideal once the down tiles can
  // make up the gate-up remainder, else within one gate-up tile
  const long long ideal = (total + P - 1) / P;
  const int n_hi = U % P;
  const bool filled = n_hi == 0 || D >= (long long)w * (P - n_hi);
  if (max_load > ideal + (filled ? 1 : w)) return 5;
  return 0;
}

int main() {
  const int Us[] = {0, 1, 5, 64, 150, 151, 152, 153, 640, 700, 2048};
  const int Ds[] = {0, 1, 7, 300, 1280, 1400, 4096};
  const int Ps[] = {1, 2, 67, 75, 134, 151, 152};
  int bad = 0;
  for (int U : Us)
    for (int D : Ds)
      for (int P : Ps)
        for (int w = 1; w <= 5; ++w) {
          const int r = check(U, D, P, w);
          if (r != 0) {
            if (bad < 10) printf("FAIL U=%d D=%d P=%d w=%d code %d\n", U, D, P, w, r);
            ++bad;
          }
        }
  printf("%s\n", bad == 0 ? "ok" : "failures");
  return bad == 0 ? 0 : 1;
}
'''


def test_fused_schedule_covers_orders_and_balances(tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    src = tmp_path / "sched.cu"
    src.write_text(PROGRAM)
    exe = tmp_path / "sched"
    subprocess.run([nvcc, "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True,
                   capture_output=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout
