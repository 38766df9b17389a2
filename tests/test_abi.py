"""The C-ABI library builds, loads without a GPU and exports every entry
point declared in include/*.h (no compute calls: this runs on CPU)."""
import ctypes
import glob
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names.update(re.findall(r"\b(ro_\w+)\s*\(", src))
    return sorted(names)


def test_library_exports_every_declared_entry_point():
    from paper_2609_18703_gb300 import build
    lib_path = build.build()
    lib = ctypes.CDLL(lib_path)
    names = declared_symbols()
    assert "ro_expand" in names and "ro_assemble" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_abi():
    import paper_2609_18703_gb300 as pkg
    assert set(declared_symbols()) <= set(pkg.EXPORTS)
    for n in pkg.EXPORTS:
        assert callable(getattr(pkg, n))


def test_create_without_gpu_fails_cleanly():
    import torch
    if torch.cuda.is_available():
        return
    import paper_2609_18703_gb300 as pkg
    h = ctypes.c_void_p()
    st = pkg.load().ro_ctx_create(ctypes.byref(h), 0, None, 1)
    assert st == pkg.RO_E_CUDA and not h.value


def test_binding_kernel_names_follow_the_header_ids():
    """The binding's kernel names (profiling) are the header's RO_K_* ids in order."""
    from paper_2609_18703_gb300._binding import KERNELS
    src = open(os.path.join(ROOT, "include", "rayorch_gpu.h")).read()
    block = re.search(r"enum \{\s*(RO_K_EXPAND_SCAN.*?)\};", src, re.S).group(1)
    ids = {n: int(v) for n, v in re.findall(r"RO_K_(\w+)\s*=\s*(\d+)", block)}
    count = ids.pop("COUNT")
    assert sorted(ids.values()) == list(range(count))
    assert [n.lower() for n, _ in sorted(ids.items(), key=lambda kv: kv[1])] == list(KERNELS)
