"""Host-side checks of the C ABI: the library builds for sm_103a, loads without a GPU,
exports every function include/stacklstm.h declares, and rejects bad arguments before
touching a device."""
import ctypes

import pytest

from paper_1904_03409_gb300 import binding, build


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.load()


def test_exports_every_declared_function(lib):
    names = binding.header_functions()
    assert {"stacklstm_create", "stacklstm_forward", "stacklstm_backward", "stacklstm_destroy",
            "stacklstm_status_string"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(lib):
    for code in range(9):
        assert lib.stacklstm_status_string(code).decode() not in ("", "unknown status")
    assert lib.stacklstm_status_string(99).decode() == "unknown status"


@pytest.mark.parametrize("T,B,I,H,dt", [(0, 1, 1, 1, 0), (1, 0, 1, 1, 0), (1, 1, 0, 1, 0), (1, 1, 1, 0, 0),
                                        (1, 1, 1, 1, 7)])
def test_create_rejects_bad_sizes(lib, T, B, I, H, dt):
    h = ctypes.c_void_p()
    assert lib.stacklstm_create(ctypes.byref(h), T, B, I, H, dt, 0, None) == 1
    assert h.value is None


def test_create_rejects_unsupported_bf16_shapes(lib):
    h = ctypes.c_void_p()
    # the bf16 path moves rows in 16-byte pieces: I and H must be multiples of 8
    assert lib.stacklstm_create(ctypes.byref(h), 4, 4, 12, 16, 1, 0, None) == 7
    assert lib.stacklstm_create(ctypes.byref(h), 4, 4, 16, 20, 1, 0, None) == 7


def test_null_handle(lib):
    assert lib.stacklstm_forward(*([None] * 13)) == 1
    assert lib.stacklstm_backward(*([None] * 8)) == 1
    assert lib.stacklstm_status(None) == 1
    assert lib.stacklstm_destroy(None) == 0
    assert lib.stacklstm_create(None, 1, 1, 1, 1, 0, 0, None) == 1


def test_binding_refuses_without_library(tmp_path):
    saved = binding._lib
    binding._lib = None
    try:
        with pytest.raises(RuntimeError):
            binding.load(str(tmp_path / "missing.so"))
    finally:
        binding._lib = saved


@pytest.mark.parametrize("T,Tb,B,H,P,A,want", [(0, 4, 2, 8, 8, 3, 1), (4, 0, 2, 8, 8, 3, 1), (4, 4, 0, 8, 8, 3, 1),
                                               (4, 4, 2, 0, 8, 3, 1), (4, 4, 2, 8, 0, 3, 1), (4, 4, 2, 8, 8, 1, 1),
                                               (4, 4, 2, 12, 8, 3, 7), (4, 4, 2, 8, 300, 3, 7),
                                               (4, 4, 2, 8, 8, 9, 7)])
def test_head_create_rejects_bad_sizes(lib, T, Tb, B, H, P, A, want):
    # the parser head: H a multiple of 8, state width <= 256, 2..8 transitions
    h = ctypes.c_void_p()
    assert lib.stacklstm_head_create(ctypes.byref(h), T, Tb, B, H, P, A, 0, None) == want
    assert h.value is None


def test_head_null_handle(lib):
    assert lib.stacklstm_head_create(None, 4, 4, 2, 8, 8, 3, 0, None) == 1
    assert lib.stacklstm_head_run(*([None] * 21)) == 1
    assert lib.stacklstm_head_add_h0_grads(None, None, None) == 1
    assert lib.stacklstm_head_status(None) == 1
    assert lib.stacklstm_head_destroy(None) == 0
    assert lib.stacklstm_head_last_error(None).decode() == "null handle"
