"""The boundary is usable from plain C.

A small C11 program, compiled with the system C compiler against
include/w8a8.h alone and linked with the built library, calls entry points
whose argument checks fail on the host (so no device is touched) and the
host-only helpers, and prints their results.  It proves that the header is
valid C (not only C++) and that the exported symbols resolve from C.
"""

import os
import shutil
import subprocess

import pytest

from paper_2606_12280_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stdio.h>
#include <stdint.h>
#include "w8a8.h"

int main(void) {
    /* host-only helpers */
    printf("%s\n", w8a8_status_string(W8A8_ERR_MISALIGNED));
    printf("%lld\n", w8a8_chunk_plan_size(12288, 4096));
    /* argument checks fail on the host: nothing reaches a device */
    uintptr_t a = 0x100000;
    int8_t *Xq = (int8_t *)a, *Wq = (int8_t *)(a + 0x1000);
    float *s = (float *)(a + 0x2000);
    uint16_t *Y = (uint16_t *)(a + 0x3000);
    printf("%d\n", (int)w8a8_linear(Xq, s, Wq, s, 0, 16, 8, 15, Y, 0, 0, 0));    /* K % 16 != 0 */
    printf("%d\n", (int)w8a8_linear(Xq, s, Wq, s, 0, 16, 8, 16, (uint16_t *)(a + 2), 0, 0, 0)); /* misaligned */
    printf("%d\n", (int)w8a8_quant_act(0, 0, 4, 16, Xq, s, 0));                   /* null X */
    printf("%d\n", (int)w8a8_linear(Xq, s, Wq, s, 0, 0, 8, 16, Y, 0, 0, 0));     /* M == 0: no-op */
    return 0;
}
"""


def test_header_compiles_and_links_as_c(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lib = _build.build()
    src = tmp_path / "use_w8a8.c"
    src.write_text(PROGRAM)
    exe = tmp_path / "use_w8a8"
    subprocess.run([cc, "-std=c11", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src),
                    "-o", str(exe), lib, "-Wl,-rpath," + os.path.dirname(lib)], check=True,
                   capture_output=True, text=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()
    assert out[0] == "W8A8_ERR_MISALIGNED"
    assert int(out[1]) == 48 * 2             # 48 blocks of 256 rows, one bit word + one max word each
    assert out[2:] == ["2", "3", "1", "0"]
