"""The C-ABI library loads on a machine without a GPU and exports every entry
point that include/*.h declares (no compute calls here)."""
import ctypes
import glob
import os
import re

from paper_2608_15438_gb300 import neuroute as nr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(nr_\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return names


def test_every_declared_symbol_is_exported():
    names = declared_functions()
    assert {"nr_index_load", "nr_encode", "nr_route", "nr_search"} <= names
    L = ctypes.CDLL(nr.LIB_PATH)
    for n in sorted(names):
        assert hasattr(L, n), n
    assert names <= set(nr.EXPORTS)


def test_host_only_calls():
    L = nr.lib()
    assert L.nr_status_string(-6) == b"NR_ERR_DEVICE_CHECK"
    assert L.nr_status_string(0) == b"NR_OK"
    p = nr.params()
    assert (p.round_size, p.t_low, p.u_min, p.f_min, p.r_min) == (256, 4, 1, 1, 1)
    assert p.alpha_front == 0.5 and p.gate_m0 == float("inf")
    # bad arguments are rejected before any device work
    assert L.nr_index_load(None, 0, None) == -1
    assert L.nr_set_params(None, None) == -1
    assert L.nr_search(None, None, 0, 10, 8, 32, None, None, None) == -1
    assert L.nr_kernel_launches(None) == 0
