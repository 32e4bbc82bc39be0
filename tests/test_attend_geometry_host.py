"""The attention pass's chunk geometry (make_geom, decode_chunk in csrc/lg_attend_mma.cu),
compiled for the host from the kernel's own source text, over a sweep of shapes: chunk rows a
multiple of the 128-row tile, never more chunks per (layer, sequence, kv-head) group than the
workspace holds (its partials would overrun it), every row of the longest group covered, no
empty chunk, and chunk ids mapping one to one onto (layer, sequence, kv-head, chunk)."""
import os
import re
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "paper_2604_10044_gb300", "csrc", "lg_attend_mma.cu")


def _block(text, start_pat):
    """the text from start_pat's match to its closing brace (and a following ';' for a struct)"""
    m = re.search(start_pat, text, flags=re.M)
    assert m, start_pat
    i = text.index("{", m.start())
    depth = 0
    for j in range(i, len(text)):
        depth += {"{": 1, "}": -1}.get(text[j], 0)
        if depth == 0:
            end = j + 1
            if text[end:end + 1] == ";":
                end += 1
            return text[m.start():end]
    raise AssertionError("unbalanced " + start_pat)


HARNESS = r'''
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <random>
#include <set>
#include <tuple>
#define __device__
#define __forceinline__ inline
static inline int max(int a, int b) { return a > b ? a : b; }
static inline unsigned max(unsigned a, unsigned b) { return a > b ? a : b; }
static inline int min(int a, int b) { return a < b ? a : b; }
struct AttendArgs { int H_kv, n_layers, batch, max_chunks; };
%(consts)s
%(structs)s
%(funcs)s
static int fails = 0;
#define CHECK(c, ...) do { if (!(c) && fails++ < 10) { std::printf(__VA_ARGS__); std::printf("\n"); } } while (0)
static void one(int H_kv, int L, int b, int max_chunks, int n_max, long long len_sum, bool ids) {
  AttendArgs a{H_kv, L, b, max_chunks};
  const Geom g = make_geom(a, n_max, len_sum, 152);
  CHECK(g.rows >= kTile && g.rows %% kTile == 0, "rows %%d", g.rows);
  CHECK(g.per_grp >= 1 && g.per_grp <= max_chunks, "per_grp %%d of %%d (n %%d)", g.per_grp, max_chunks, n_max);
  CHECK((long long)g.per_grp * g.rows >= n_max, "coverage %%d x %%d < %%d", g.per_grp, g.rows, n_max);
  CHECK((long long)(g.per_grp - 1) * g.rows < n_max, "empty last chunk %%d x %%d, n %%d", g.per_grp, g.rows, n_max);
  CHECK(g.groups == L * b * H_kv && g.total == g.groups * g.per_grp, "totals");
  if (ids) {
    std::set<std::tuple<int, int, int, int>> seen;
    for (int c = 0; c < g.total; ++c) {
      const ChunkId id = decode_chunk(a, c, g);
      CHECK(id.lloc >= 0 && id.lloc < L && id.b >= 0 && id.b < b && id.kvh >= 0 && id.kvh < H_kv &&
            id.ch >= 0 && id.ch < g.per_grp, "id out of range");
      seen.insert(std::make_tuple(id.lloc, id.b, id.kvh, id.ch));
    }
    CHECK((int)seen.size() == g.total, "ids not one to one");
  }
}
int main() {
  // the benchmark's shapes: the paper's setting (28 layers, 8 kv-heads, b 1, 960..1024 rows,
  // 2 chunks of 512 rows: 448 chunks, at least 3 a CTA on 152 CTAs)
  for (int n = 960; n <= 1024; ++n) {
    AttendArgs a{8, 28, 1, 16};
    const Geom g = make_geom(a, n, n, 152);
    CHECK(g.per_grp == 2 && g.rows == 512, "paper shape n %%d: %%d x %%d", n, g.per_grp, g.rows);
  }
  std::mt19937_64 rng(1);
  auto pick = [&](long long lo, long long hi) { return lo + (long long)(rng() %% (unsigned long long)(hi - lo + 1)); };
  const int hk[] = {1, 2, 4, 8}, ls[] = {1, 2, 28, 32};
  for (int it = 0; it < 60000; ++it) {
    const int H_kv = hk[pick(0, 3)], L = ls[pick(0, 3)], b = (int)pick(1, 64);
    const int max_chunks = (int)pick(1, 64);
    const int n_max = (int)pick(1, it %% 2 ? 140000 : 5000);
    const long long len_sum = pick(n_max, (long long)n_max * b);
    one(H_kv, L, b, max_chunks, n_max, len_sum, (long long)L * b * H_kv * max_chunks <= 4096);
  }
  std::printf("mismatches %%d\n", fails);
  return fails != 0;
}
'''


def test_attend_geometry_invariants():
    if shutil.which("g++") is None:
        pytest.skip("needs g++")
    text = open(SRC).read()
    consts = "\n".join(re.findall(r"^constexpr int (?:kTile|kMaxChunkRows) = [^;]+;", text, flags=re.M))
    assert "kTile" in consts and "kMaxChunkRows" in consts
    structs = _block(text, r"^struct ChunkId \{") + "\n" + _block(text, r"^struct Geom \{")
    funcs = (_block(text, r"^__device__ __forceinline__ Geom make_geom\(") + "\n" +
             _block(text, r"^__device__ __forceinline__ ChunkId decode_chunk\("))
    src = HARNESS % dict(consts=consts, structs=structs, funcs=funcs)
    with tempfile.TemporaryDirectory() as d:
        cpp, exe = os.path.join(d, "geom.cpp"), os.path.join(d, "geom")
        open(cpp, "w").write(src)
        subprocess.run(["g++", "-O2", "-std=c++17", cpp, "-o", exe], check=True)
        r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout
