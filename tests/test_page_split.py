"""The page split shared by the tensor-core decode kernels (`csrc/lla_units.cuh`), compiled for
the host and checked exhaustively on the CPU: CTA c of `grid` holds the global pages
[page_lo(c), page_lo(c + 1)); the ranges tile [0, np) in order, differ in length by at most one,
and cta_of(g) names the CTA whose range holds page g.  The attention kernels cut the batch's
pages with page_lo; the finish kernels find a unit's runs (the CTAs from cta_of(first page) to
cta_of(last page)) with cta_of, so a disagreement would merge the wrong partials."""
import os
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_15456_gb300", "csrc")

CHECK = r"""
#include <cstdio>
#include <cstdint>
#include "lla_units.cuh"

static int fails = 0;
static void fail(const char *what, int64_t np, int grid, int64_t x) {
    if (fails++ < 10) std::printf("%s np=%lld grid=%d at %lld\n", what, (long long)np, grid, (long long)x);
}

static void check(int np, int grid) {
    using lla::page_lo;
    using lla::cta_of;
    if (page_lo(0, np, grid) != 0) fail("first", np, grid, 0);
    if (page_lo(grid, np, grid) != np) fail("last", np, grid, grid);
    const int lo = np / grid, hi = (np + grid - 1) / grid;
    for (int c = 0; c < grid; ++c) {
        const int n = page_lo(c + 1, np, grid) - page_lo(c, np, grid);
        if (n < lo || n > hi) fail("range length", np, grid, c);
    }
    for (int g = 0; g < np; ++g) {
        const int c = cta_of(g, np, grid);
        if (c < 0 || c >= grid || page_lo(c, np, grid) > g || g >= page_lo(c + 1, np, grid))
            fail("cta_of", np, grid, g);
    }
}

int main() {
    for (int grid = 1; grid <= 1024; grid += (grid < 300 ? 1 : 37))
        for (int np = 0; np <= 700; ++np) check(np, grid);
    // batch sizes of the benchmark workloads (pages of one call) and large counts, at the
    // grids of GB300 (152 SMs) and of the largest supported launch
    const int big[] = {860, 13760, 42403, 1 << 20, (1 << 20) + 7};
    for (int np : big)
        for (int grid : {1, 7, 148, 152, 256, 1024}) check(np, grid);
    // page_lo's product stays in 64 bits near the 32-bit page limit
    const int np = 2147483647;
    for (int grid : {152, 1024})
        for (int c = 0; c <= grid; ++c) {
            const int64_t want = static_cast<int64_t>(c) * np / grid;
            if (lla::page_lo(c, np, grid) != want) fail("large page_lo", np, grid, c);
        }
    std::printf("%s\n", fails ? "FAILED" : "ok");
    return fails ? 1 : 0;
}
"""


def test_page_split_tiles_the_pages_and_cta_of_inverts_it():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not available")
    with tempfile.TemporaryDirectory() as tmp:
        src = os.path.join(tmp, "page_split_check.cu")
        exe = os.path.join(tmp, "page_split_check")
        with open(src, "w") as f:
            f.write(CHECK)
        r = subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O2", "-std=c++17",
                            "-I", CSRC, "-I", os.path.join(ROOT, "include"), src, "-o", exe],
                           capture_output=True, text=True)
        assert r.returncode == 0, r.stderr[-3000:]
        r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
        assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout[-2000:]
