"""The C ABI from C: a small C99 program includes include/blr.h, links against
libblr.so and calls the host-only entry points (sizing, kernel family, status
text, argument validation). Nothing reaches the GPU."""
import os
import shutil
import subprocess

import pytest

from paper_2406_12580_gb300 import _lib
from paper_2406_12580_gb300 import build as blr_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "blr.h"

int main(void) {
  blr_desc headline = {256, 200, 64, BLR_F32, 1.0f};
  blr_desc longseq = {8, 32768, 512, BLR_BF16, 1.0f};
  blr_desc bad = {2, 10, 12, BLR_F32, 1.0f};
  printf("ws %zu %zu %zu\n", blr_workspace_bytes(&headline), blr_workspace_bytes(&longseq),
         blr_workspace_bytes(&bad));
  printf("family %d %d %d %d\n", blr_scan_family(&headline, 0), blr_scan_family(&longseq, 0),
         blr_scan_family(&longseq, 1), blr_scan_family(&bad, 0));
  printf("status %s\nstatus %s\n", blr_status_string(BLR_OK), blr_status_string(BLR_ERR_UNSUPPORTED));
  /* D not a multiple of 8: refused on the host, nothing enqueued */
  blr_status s = blr_scan_fwd(&bad, NULL, NULL, NULL, NULL, NULL, NULL, NULL, 0, NULL);
  printf("fwd %d %s\n", (int)s, strstr(blr_last_error_string(), "multiple of 8") ? "msg" : "nomsg");
  return 0;
}
"""


def test_c_client_links_and_calls_host_entry_points(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    if blr_build.stale():
        blr_build.build()
    lib_dir = os.path.dirname(_lib.library_path())
    src = tmp_path / "client.c"
    exe = tmp_path / "client"
    src.write_text(C_CLIENT)
    subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src),
                    "-L", lib_dir, "-lblr", f"-Wl,-rpath,{lib_dir}", "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], stdout=subprocess.PIPE, text=True, check=True).stdout.split("\n")
    ws = [int(v) for v in out[0].split()[1:]]
    assert ws[0] > 0 and ws[1] > ws[0] and ws[2] == 0
    assert out[1].split()[1:] == ["2", "3", "1", "0"]  # serial, segmented, tiled (lengths), none
    assert out[2].startswith("status BLR_OK") and out[3].startswith("status BLR_ERR_UNSUPPORTED")
    assert out[4] == f"fwd {_lib.BLR_ERR_UNSUPPORTED} msg"
