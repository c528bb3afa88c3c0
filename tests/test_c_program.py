"""The library from plain C: a C99 program that includes only include/flarepp.h and links
libflarepp.so sizes a workspace, reads the status strings and has bad arguments rejected. No
call here reaches the GPU, so it runs without one; it shows that the boundary needs neither
C++ nor PyTorch."""
import os
import shutil
import subprocess

import pytest

from paper_2608_11519_gb300 import build as lib_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "flarepp.h"

static int fails = 0;
#define CHECK(c) do { if (!(c)) { printf("FAILED: %s (line %d)\n", #c, __LINE__); ++fails; } } while (0)

int main(void) {
    flarepp_shape s = {1, 8, 1048576, 512, 32, FLAREPP_BF16};
    size_t ws = flarepp_route_workspace_bytes(&s);
    CHECK(ws > 0 && ws % 256 == 0);
    CHECK(flarepp_route_workspace_bytes(NULL) == 0);
    flarepp_shape bad = s;
    bad.D = 48;
    CHECK(flarepp_route_workspace_bytes(&bad) == 0);
    CHECK(flarepp_route_saved_bytes(&s) > 0);
    CHECK(flarepp_route_host_buffer_bytes(&s) >= 5 * (size_t)8 * 1048576 * 32 * 2);
    CHECK(flarepp_mixer_workspace_bytes(&s, 4) > flarepp_mixer_workspace_bytes(&s, 2));
    CHECK(strcmp(flarepp_status_string(FLAREPP_OK), "ok") == 0);
    CHECK(strlen(flarepp_version()) > 0);
    /* rejected before any CUDA call: unsupported D, a null K, a non-finite scale */
    char* base = (char*)(uintptr_t)0x7F0000000000ull;
    const size_t step = (size_t)1 << 36;
    CHECK(flarepp_route_fwd(&bad, base, base + step, base + 2 * step, base + 3 * step,
                            base + 4 * step, 0.25f, base + 5 * step, base + 6 * step, ws, NULL)
          == FLAREPP_ERR_UNSUPPORTED);
    CHECK(flarepp_route_fwd(&s, base, base + step, base + 2 * step, NULL, base + 4 * step, 0.25f,
                            base + 5 * step, base + 6 * step, ws, NULL)
          == FLAREPP_ERR_INVALID_ARGUMENT);
    float inf = 1e30f;
    inf = inf * inf;
    CHECK(flarepp_route_fwd(&s, base, base + step, base + 2 * step, base + 3 * step,
                            base + 4 * step, inf, base + 5 * step, base + 6 * step, ws, NULL)
          == FLAREPP_ERR_INVALID_ARGUMENT);
    /* an empty problem is a successful no-op */
    flarepp_shape empty = s;
    empty.B = 0;
    CHECK(flarepp_route_fwd(&empty, NULL, NULL, NULL, NULL, NULL, 0.25f, NULL, NULL, 0, NULL)
          == FLAREPP_OK);
    printf("%s\n", fails ? "failed" : "ok");
    return fails != 0;
}
"""


@pytest.mark.skipif(shutil.which("gcc") is None, reason="no C compiler")
def test_plain_c_program_uses_the_abi(tmp_path):
    lib_build.build()
    lib = lib_build.lib_path()
    src = tmp_path / "abi.c"
    src.write_text(PROGRAM)
    exe = tmp_path / "abi"
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-pedantic", "-I",
                    os.path.join(ROOT, "include"), str(src), "-o", str(exe), "-L",
                    os.path.dirname(lib), "-l:" + os.path.basename(lib),
                    "-Wl,-rpath," + os.path.dirname(lib)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr
