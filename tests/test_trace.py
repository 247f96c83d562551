"""NVTX ranges around the C-ABI calls, checked without a GPU.

A tiny NVTX injection library (compiled here with gcc) takes the place of a
profiler: loaded through NVTX_INJECTION64_PATH, it records the name of every
range the library pushes.  A fresh process (NVTX reads the variable once, at
the first range of a process) calls host-only entry points and a call that is
rejected before any CUDA work, then reads the record back.
"""
import os
import shutil
import subprocess
import sys
import textwrap

import pytest

from paper_1911_08020_gb300 import build as darb_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

INJECTION = r"""
#include <stddef.h>
#include <stdint.h>
#include <string.h>
typedef void (*fn_t)(void);
typedef fn_t **table_t;
typedef struct { size_t struct_size; int (*get_module)(int module, table_t *out, unsigned *size); } callbacks_t;
typedef const void *(*get_export_t)(uint32_t id);
static char buf[1 << 16];
static size_t len;
static int depth;
static int push(const char *name) {
    size_t n = strlen(name);
    if (len + n + 2 < sizeof buf) { memcpy(buf + len, name, n); len += n; buf[len++] = '\n'; }
    return depth++;
}
static int pop(void) { return --depth; }
const char *trace_record(void) { buf[len] = 0; return buf; }
int trace_depth(void) { return depth; }
/* NVTX asks the injection for its callbacks: export table 1 (callbacks),
   module 1 (core), slots 9 (RangePushA) and 11 (RangePop). */
int InitializeInjectionNvtx2(get_export_t get) {
    const callbacks_t *cb = (const callbacks_t *)get(1);
    table_t table = 0;
    unsigned size = 0;
    if (!cb || !cb->get_module(1, &table, &size) || !table || size <= 11) return 0;
    *table[9] = (fn_t)push;
    *table[11] = (fn_t)pop;
    return 1;
}
"""

CHILD = textwrap.dedent("""
    import ctypes, sys
    import numpy as np
    sys.path.insert(0, sys.argv[1])
    from paper_1911_08020_gb300 import darb
    L = darb.lib()
    nnz = np.array([12, 6, 5, 5], dtype=np.int64)
    m = np.zeros(4, dtype=np.int32)
    assert L.darb_assign_block_sizes(nnz.ctypes.data, 4, 32, 1, 256, m.ctypes.data) == darb.OK
    assert L.darb_spmm(None, None, 1, 1, None, 1, None) == darb.ERR_INVALID_ARG
    rec = ctypes.CDLL(sys.argv[2])
    rec.trace_record.restype = ctypes.c_char_p
    print(rec.trace_record().decode(), end="")
    print("depth", rec.trace_depth())
""")


def test_c_abi_calls_are_nvtx_ranges(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    darb_build.build()
    src = tmp_path / "inject.c"
    src.write_text(INJECTION)
    lib = tmp_path / "libinject.so"
    subprocess.run([cc, "-O1", "-fPIC", "-shared", str(src), "-o", str(lib)], check=True)
    env = dict(os.environ, NVTX_INJECTION64_PATH=str(lib))
    out = subprocess.run([sys.executable, "-c", CHILD, ROOT, str(lib)], env=env, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    lines = out.stdout.splitlines()
    assert lines[-1] == "depth 0"                       # every range was closed
    names = lines[:-1]
    assert names == ["darb_assign_block_sizes", "darb_spmm", "darb_spmm_ex"], names
