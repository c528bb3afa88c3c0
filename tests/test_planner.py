"""The tensor-core encode's chunk plan on the host: make_plan (plan.cu, compiled here as host
code) against an exhaustive search of the same cost model. make_plan tries only the largest
chunk count of each wave count and stops at a lower bound on the cost; this checks that it
still returns the minimiser an exhaustive search finds, and that its chunks cover the tokens in
whole items. No GPU is used: the planner is plain host code."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_11519_gb300", "csrc")

HARNESS = r"""
#include <stdio.h>
#include <random>
#include "flarepp_internal.h"

// tokens per encode item and routes per group, as the tensor-core encode defines them
namespace flarepp {
int64_t tc_encode_item_rows(int64_t D) { return D == 64 ? 64 : (D == 16 ? 112 : 96); }
int64_t tc_group_rows(int64_t D) { (void)D; return 512; }
}  // namespace flarepp

using flarepp::cdiv;

// the exhaustive search: every chunk count n, cost = waves x (items x na / ns + 3), the
// smallest n of least cost
static int64_t exhaustive_chunk_len(int64_t BH, int64_t N, int64_t M, int64_t D) {
    const int64_t item = flarepp::tc_encode_item_rows(D), group = flarepp::tc_group_rows(D);
    const int64_t ns = group / 128, n_groups = cdiv(M, group);
    const int64_t tiles0 = M >= group ? ns : cdiv(M, 128);
    const double na = tiles0 <= 1 ? 1.0 : (tiles0 <= 2 ? 2.0 : 4.0);
    const int64_t per_chunk = BH * n_groups, max_chunks = cdiv(N, item);
    double best = 1e300;
    int64_t best_n = 1;
    for (int64_t n = 1; n <= max_chunks && n <= 65536; ++n) {
        const double cost = (double)cdiv(per_chunk * n, flarepp::kNumSMs) *
                            ((double)cdiv(cdiv(N, n), item) * na / (double)ns + 3.0);
        if (cost < best) {
            best = cost;
            best_n = n;
        }
    }
    return cdiv(cdiv(N, best_n), item) * item;
}

int main() {
    std::mt19937_64 g(11);
    int bad = 0, n = 0;
    auto check = [&](int64_t B, int64_t H, int64_t N, int64_t M, int64_t D) {
        flarepp_shape s{B, H, N, M, D, FLAREPP_BF16};
        flarepp::Plan p;
        if (flarepp::make_plan(&s, &p) != FLAREPP_OK) return;
        ++n;
        const int64_t item = flarepp::tc_encode_item_rows(D);
        const int64_t want = exhaustive_chunk_len(B * H, N, M, D);
        const bool ok = p.chunk_len == want && p.chunk_len % item == 0 &&
                        p.nchunk == cdiv(N, p.chunk_len) && (p.nchunk - 1) * p.chunk_len < N;
        if (!ok && bad++ < 5)
            printf("mismatch B=%ld H=%ld N=%ld M=%ld D=%ld: %ld vs %ld\n", (long)B, (long)H,
                   (long)N, (long)M, (long)D, (long)p.chunk_len, (long)want);
    };
    for (int64_t B : {1, 2, 4, 16, 64})
        for (int64_t H : {1, 3, 8, 16})
            for (int64_t N : {1, 63, 64, 65, 95, 96, 97, 5000, 16384, 100000, 1 << 20, (1 << 20) + 17})
                for (int64_t M : {1, 128, 300, 512, 513, 2048})
                    for (int64_t D : {16, 32, 64}) check(B, H, N, M, D);
    for (int i = 0; i < 1500; ++i)
        check(1 + g() % 64, 1 + g() % 16, 1 + g() % (1 << 21), 1 + g() % 2048, 16 << (g() % 3));
    printf("%d shapes, %d mismatches\n", n, bad);
    return bad != 0;
}
"""


@pytest.mark.skipif(shutil.which("nvcc") is None, reason="nvcc not found")
def test_pruned_chunk_search_matches_exhaustive_search(tmp_path):
    src = tmp_path / "plan_check.cu"
    src.write_text(HARNESS)
    exe = tmp_path / "plan_check"
    subprocess.run(["nvcc", "-std=c++17", "-O2", "-I", CSRC, "-I", os.path.join(ROOT, "include"),
                    str(src), os.path.join(CSRC, "plan.cu"), "-o", str(exe)], check=True,
                   capture_output=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert " 0 mismatches" in r.stdout
