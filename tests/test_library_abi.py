"""CPU-side checks of the C ABI: the library builds, loads without a GPU, and exports
every entry point that include/mure.h declares; the binding's structures have the
header's layout; host-side validation needs no device."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "mure.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mure_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def libpath():
    from paper_2607_18582_gb300 import build
    return build.build()


def test_library_exports_every_declared_symbol(libpath):
    names = declared_functions()
    assert len(names) >= 12
    lib = ctypes.CDLL(libpath)  # loads on a machine without a GPU
    for n in names:
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (mure_\w+)", out))
    assert set(names) <= exported
    from paper_2607_18582_gb300 import mure
    assert set(mure.EXPORTS) == set(names)


def _c_layout(tmp_path, struct, fields):
    """sizeof and offsetof of a header struct, printed by a C program compiled against
    include/mure.h with gcc."""
    src = tmp_path / f"{struct}.c"
    body = "".join(f'    printf("%zu\\n", offsetof({struct}, {f}));\n' for f in fields)
    src.write_text(f'#include <stddef.h>\n#include <stdio.h>\n#include "mure.h"\nint main(void) {{\n'
                   f'    printf("%zu\\n", sizeof({struct}));\n{body}    return 0;\n}}\n')
    exe = tmp_path / f"{struct}.bin"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)], check=True)
    vals = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    return vals[0], vals[1:]


def test_struct_layouts_match_header(tmp_path):
    from paper_2607_18582_gb300 import mure
    for struct, cls in (("mure_node", mure._Node), ("mure_model_desc", mure._ModelDesc),
                        ("mure_allocator", mure._Allocator), ("mure_eval_opts", mure._Opts),
                        ("mure_eval_stats", mure._Stats)):
        names = [f for f, _ in cls._fields_]
        size, offs = _c_layout(tmp_path, struct, names)
        assert ctypes.sizeof(cls) == size, struct
        assert [getattr(cls, f).offset for f in names] == offs, struct
    size, offs = _c_layout(tmp_path, "mure_mutant", list(mure.MUTANT_DTYPE.names))
    assert mure.MUTANT_DTYPE.itemsize == size
    assert [mure.MUTANT_DTYPE.fields[f][1] for f in mure.MUTANT_DTYPE.names] == offs


def test_library_loads_and_fails_cleanly_without_gpu(libpath):
    """With no usable device, context creation returns an error status (it never
    falls back to the CPU)."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2607_18582_gb300 import mure
    out = ctypes.c_void_p()
    st = mure.lib().mure_create(0, None, None, ctypes.byref(out))
    assert st != 0 and not out.value
