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


def test_struct_layouts_match_header():
    from paper_2607_18582_gb300 import mure
    assert ctypes.sizeof(mure._Node) == 10 * 4 + 2 * 8
    assert mure.MUTANT_DTYPE.itemsize == 40
    assert mure.MUTANT_DTYPE.fields["neuron_off"][1] == 16
    assert mure.MUTANT_DTYPE.fields["seed"][1] == 32
    assert ctypes.sizeof(mure._Opts) == 24
    assert ctypes.sizeof(mure._Stats) == 4 * 8 + 6 * 8 + 64 * 8 * 3 + 3 * 8 + 3 * 8


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
