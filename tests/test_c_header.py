"""include/gemmi.h is a plain C header: a C99 program that includes it, takes the address of every
function it declares and links against the library builds with warnings as errors, and runs the
host-side calls that need no GPU (argument checks, options, empty problems, the version string).
"""
import os
import re
import shutil
import subprocess
import tempfile

import pytest

import paper_2302_07594_gb300 as gm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gemmi.h")


def declared_functions():
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*([a-z_0-9]+)\s*\(", text, flags=re.M)
    return sorted(set(n for n in names if n not in ("if", "while")))


PROGRAM = r'''
#include <stdio.h>
#include <string.h>
#include "gemmi.h"

static void* const every_function[] = { %(ptrs)s };

int main(void) {
  int rc;
  if (sizeof(every_function) / sizeof(every_function[0]) != %(count)d) return 10;
  /* an empty problem is a no-op that touches no device */
  if (gemm_i16(0, 4, 4, NULL, 4, NULL, 4, NULL, 4) != GEMMI_OK) return 11;
  /* a negative dimension is refused on the host, with a message */
  rc = gemm_i8(-1, 4, 4, NULL, 4, NULL, 4, NULL, 4);
  if (rc != GEMMI_EINVAL || strlen(gemmi_last_error()) == 0) return 12;
  /* options round-trip */
  if (gemmi_set_option(GEMMI_OPT_TC_CHUNK_SCALE, 1) != GEMMI_OK) return 13;
  if (gemmi_get_option(GEMMI_OPT_TC_CHUNK_SCALE) != 1) return 14;
  if (gemmi_set_option(GEMMI_OPT_TC_CHUNK_SCALE, 3) != GEMMI_EINVAL) return 15;
  if (gemmi_set_option(GEMMI_OPT_TC_CHUNK_SCALE, 2) != GEMMI_OK) return 16;
  printf("%%s\n", gemmi_version());
  return 0;
}
'''


def test_header_compiles_links_and_runs_as_c99():
    if shutil.which("gcc") is None:
        pytest.skip("gcc is not installed")
    gm.build()
    names = declared_functions()
    src = PROGRAM % {"ptrs": ", ".join(f"(void*)&{n}" for n in names), "count": len(names)}
    libdir = os.path.dirname(gm.LIB_PATH)
    with tempfile.TemporaryDirectory() as d:
        c, exe = os.path.join(d, "use_gemmi.c"), os.path.join(d, "use_gemmi")
        with open(c, "w") as f:
            f.write(src)
        # function-to-object pointer casts are outside ISO C; everything else is held to C99
        r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
                            c, "-o", exe, "-L", libdir, "-lgemmi", f"-Wl,-rpath,{libdir}"],
                           capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
        r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
        assert r.returncode == 0, (r.returncode, r.stdout, r.stderr)
        assert "sm_103a" in r.stdout
