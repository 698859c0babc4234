"""The flat work plan's cost arithmetic (csrc/attn.cu), compiled for the host.

The attention kernel's flat plan lays every (sequence, kv-head) pair's items
end to end in cost units (a packed block 1, a window chunk cw, a pair's first
item sc more, the block a decode step pushes out of the window fu more) and
cuts the units into equal ranges, one per virtual warp; an item belongs to the
warp whose range holds its first unit.  The helpers are __host__ __device__,
so this test builds them with the host compiler and checks, on random shapes:

* items_below(x) counts exactly the items whose first unit item_unit(i) lies
  below x, for every item boundary, with and without flush units;
* every item costs at least 1 and at most max_item_cost units, and all items
  start inside the pair's cost;
* flat_grid's virtual-warp ranges cover [0, N) without gaps, each at least
  max_item_cost units long, and unit_owner agrees with v_first_unit.
"""

import re
import shutil
import subprocess
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]
ATTN = ROOT / "paper_2607_16248_gb300" / "csrc" / "attn.cu"

HARNESS = r"""
#include <algorithm>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
using std::max;
using std::min;
#define __host__
#define __device__
constexpr int kGroup = 32;
constexpr int kWarps = 16;
inline int packed_len(int L, int residual) {
  const int over = L - residual;
  return over > 0 ? (over / kGroup) * kGroup : 0;
}
%s
static unsigned long long rng = 88172645463325252ULL;
static unsigned long long next() { rng ^= rng << 13; rng ^= rng >> 7; rng ^= rng << 17; return rng; }
#define CHECK(c) do { if (!(c)) { printf("FAIL line %%d\n", __LINE__); return 1; } } while (0)
int main() {
  const Costs picks[3] = {{4, 1, 12}, {2, 1, 6}, {1, 0, 0}};
  long items = 0, grids = 0;
  for (int it = 0; it < 300000; ++it) {
    const Costs k = picks[it %% 3];
    const int R = (it %% 5 == 0) ? 32 : 128;
    const int L0 = (int)(next() %% 5000);
    const int L = (it %% 2) ? L0 + 1 : L0;
    const PairShape s = pair_shape(L, R);
    const int f = flush_units(L0, L, R, k);
    CHECK(!(f && s.nb < 1));
    const int C = pair_cost(s, k, f), n = s.nb + s.nr;
    if (n == 0) { CHECK(C == 0); continue; }
    for (int i = 0; i < n; ++i) {
      const int u = item_unit(i, s.nb, k, f);
      const int un = i + 1 < n ? item_unit(i + 1, s.nb, k, f) : C;
      CHECK(un - u >= 1 && un - u <= max_item_cost(k));
      CHECK(items_below(u, s.nb, s.nr, k, f) == i);
      CHECK(items_below(u + 1, s.nb, s.nr, k, f) == i + 1);
      CHECK(items_below(un, s.nb, s.nr, k, f) == i + 1);
      ++items;
    }
    CHECK(items_below(C, s.nb, s.nr, k, f) == n);
    CHECK(items_below((long long)C + 977, s.nb, s.nr, k, f) == n);
  }
  for (int it = 0; it < 20000; ++it) {
    WorkSums w;
    const long long scale = (it %% 4 == 0) ? 40 : (it %% 4 == 1) ? 4000 : 400000;
    w.nb = (long long)(next() %% (unsigned long long)scale);
    w.nr = (long long)(next() %% 5000);
    w.np = 1 + (long long)(next() %% 2048);
    w.nf = (long long)(next() %% (unsigned long long)(w.np + 1));
    const int ctas = 1 + (int)(next() %% 255);
    const FlatGrid g = flat_grid(w, ctas);
    if (g.N == 0) continue;
    CHECK(g.n_v >= 1 && g.n_v <= kWarps * ctas && g.n_cta <= ctas);
    CHECK(g.N == w.nb + g.k.cw * w.nr + g.k.sc * w.np + g.k.fu * w.nf);
    long long prev = 0;
    for (int v = 0; v < g.n_v; ++v) {
      const long long a = v_first_unit(v, g), e = v_first_unit(v + 1, g);
      CHECK(a == prev);
      CHECK(e - a >= min<long long>(g.N, max_item_cost(g.k)));
      CHECK(unit_owner(a, g) == v && unit_owner(e - 1, g) == v);
      const int c = cta_of(v, g);
      CHECK(c >= 0 && c < g.n_cta && cta_first_v(c, g) <= v);
      prev = e;
    }
    CHECK(prev == g.N);
    ++grids;
  }
  printf("ok %%ld items %%ld grids\n", items, grids);
  return 0;
}
"""


def _plan_source():
    text = ATTN.read_text()
    a = text.index("struct Costs {")
    b = text.index("// Length a kernel attends")
    body = text[a:b]
    for name in ("flush_units", "pair_cost", "item_unit", "items_below", "max_item_cost",
                 "flat_grid", "unit_owner", "v_first_unit", "cta_of", "cta_first_v"):
        assert re.search(r"\b%s\(" % name, body), name
    return body


def test_flat_plan_cost_arithmetic(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    src = tmp_path / "plan.cc"
    src.write_text(HARNESS % _plan_source())
    exe = tmp_path / "plan"
    subprocess.run([cxx, "-O2", "-std=c++17", str(src), "-o", str(exe)], check=True,
                   capture_output=True, text=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stdout + out.stderr
    assert out.stdout.startswith("ok ")
