"""The C-ABI library builds, loads on a machine without a GPU and exports
every entry point that include/spike_proj.h declares.  No compute calls."""
import ctypes
import re
from pathlib import Path

import pytest

from paper_2606_03026_gb300 import _build, spikeproj

HEADER = Path(__file__).resolve().parent.parent / "include" / "spike_proj.h"


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return spikeproj.lib()


def declared_functions():
    text = HEADER.read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(spike_proj_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("spike_proj_plan", "spike_proj_decode", "spike_proj_batched",
                     "spike_proj_prefill"):
        assert required in names


def test_header_enums_match_the_binding():
    """Every enumerator of the header's enums has the binding's value."""
    text = re.sub(r"/\*.*?\*/", "", HEADER.read_text(), flags=re.S)
    found = {}
    for body in re.findall(r"typedef enum \w+ \{(.*?)\}", text, flags=re.S):
        for name, val in re.findall(r"\b(SP_\w+)\s*=\s*(\d+)", body):
            found[name] = int(val)
    assert found["SP_SPIKES_BOOL8"] == spikeproj.SP_SPIKES_BOOL8 == spikeproj.FMTS["bool8"]
    for name, val in found.items():
        assert getattr(spikeproj, name) == val, name


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert names
    for name in names:
        assert hasattr(lib, name), f"{name} not exported by {spikeproj.LIB_PATH}"
    assert set(names) == set(spikeproj._SIGNATURES), "binding and header disagree"


def test_host_only_calls(lib):
    assert spikeproj.spike_proj_abi_version() == 1
    assert "invalid" in spikeproj.spike_proj_strerror(spikeproj.SP_EINVAL)
    # argument checks return before any CUDA call
    assert lib.spike_proj_plan(None, None, 16, None, 16, 16, 1, 0, None) == spikeproj.SP_EINVAL
    h = ctypes.c_void_p()
    fake = 1 << 20                       # never dereferenced: rejected first
    assert lib.spike_proj_plan(ctypes.byref(h), fake, 16, fake, 16, 0, 1, 0, None) == \
        spikeproj.SP_ERANGE
    assert lib.spike_proj_plan(ctypes.byref(h), fake, 16, fake, 16, 131073, 1, 0, None) == \
        spikeproj.SP_ERANGE
    assert lib.spike_proj_plan(ctypes.byref(h), fake, 16, fake, 24, 64, 1, 0, None) == \
        spikeproj.SP_EALIGN                # N % 16 != 0
    assert lib.spike_proj_plan(ctypes.byref(h), fake + 8, 16, fake, 16, 64, 1, 0, None) == \
        spikeproj.SP_EALIGN                # W not 16-byte aligned
    assert lib.spike_proj_plan(ctypes.byref(h), fake, 8, fake, 16, 64, 1, 0, None) == \
        spikeproj.SP_EALIGN                # ldw < N
    assert lib.spike_proj_plan(ctypes.byref(h), fake, 16, fake, 16, 64, 1, 0x10, None) == \
        spikeproj.SP_EINVAL                # unknown flag
    assert lib.spike_proj_decode(None, fake, 0, fake, fake, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_group_create(None, None, 0, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_group_prefill(None, None, 0, 1, 16, None, None, None) == \
        spikeproj.SP_EINVAL
    assert lib.spike_proj_probe_gather(None, fake, 1, 512, fake, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_probe_gather(fake, None, 1, 512, fake, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_probe_gather(fake, fake, 1, 768, fake, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_probe_gather(fake + 4, fake, 1, 512, fake, None) == spikeproj.SP_EALIGN
    assert lib.spike_proj_dense(None, 1, 1, None) == spikeproj.SP_EINVAL
    d = spikeproj.SpDense(fake, 32, fake, fake, 32, fake, 16, 16, 32)
    assert lib.spike_proj_dense(ctypes.addressof(d), 1, 0, None) == spikeproj.SP_EINVAL   # B = 0
    d.ldw = 24
    assert lib.spike_proj_dense(ctypes.addressof(d), 1, 1, None) == spikeproj.SP_EALIGN   # ldw % 16
    d.ldw, d.W = 32, fake + 4
    assert lib.spike_proj_dense(ctypes.addressof(d), 1, 1, None) == spikeproj.SP_EALIGN   # W alignment
    assert lib.spike_proj_lif(None, fake, 64, 1, 64, 0.5, 1.0, fake, 2, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_lif(fake, fake, 64, 1, 64, 0.5, 1.0, fake, 1, None) == spikeproj.SP_EINVAL  # ld_bits
    assert lib.spike_proj_lif(fake + 2, fake, 64, 1, 64, 0.5, 1.0, fake, 2, None) == spikeproj.SP_EALIGN
    assert lib.spike_proj_lif(fake, fake, 131073, 1, 131073, 0.5, 1.0, fake, 4097, None) == \
        spikeproj.SP_ERANGE
    assert lib.spike_proj_group_decode_lif(None, fake, fake, fake, 64, 0.5, 1.0, None, 0, None,
                                           fake, 64, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_head(None, fake, 64, 1, 0.5, 16, fake, None, None, None, None, None, 0,
                               None) == spikeproj.SP_EINVAL
    h = ctypes.c_void_p()
    assert lib.spike_proj_head_create(None, fake, 64, fake, 100, 64, None) == spikeproj.SP_EINVAL
    assert lib.spike_proj_head_create(ctypes.byref(h), fake, 64, fake, 1, 64, None) == \
        spikeproj.SP_ERANGE
    assert lib.spike_proj_head_create(ctypes.byref(h), fake, 72, fake, 100, 64, None) == \
        spikeproj.SP_EALIGN
    assert lib.spike_proj_head_destroy(None) == spikeproj.SP_OK
    assert lib.spike_proj_plan_destroy(None) == spikeproj.SP_OK
    assert lib.spike_proj_group_destroy(None) == spikeproj.SP_OK


def test_missing_library_is_an_error(monkeypatch, tmp_path):
    monkeypatch.setattr(spikeproj, "LIB_PATH", tmp_path / "absent.so")
    monkeypatch.setattr(spikeproj, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        spikeproj.lib()
