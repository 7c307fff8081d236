"""Host-side checks of the C-ABI library that need no GPU: it builds for
sm_103a, loads, exports every function include/specflash_verify.h declares,
and rejects invalid arguments before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2505_12728_gb300 import build_lib
from paper_2505_12728_gb300 import specflash_verify as sfv

HEADER = os.path.join(build_lib.ROOT, "include", "specflash_verify.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(sf_\w+)\s*\(", text, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    build_lib.build()
    return sfv.load_library()


def test_header_declares_the_binding_symbols():
    assert declared_functions() == sorted(sfv.EXPORTED_SYMBOLS)


def test_library_exports_every_declared_function(lib):
    raw = ctypes.CDLL(build_lib.LIB)
    for name in declared_functions():
        assert hasattr(raw, name), f"{name} not exported"


def test_status_strings_and_version(lib):
    assert lib.sf_status_string(0) == b"SF_OK"
    assert lib.sf_status_string(1) == b"SF_ERR_INVALID_ARG"
    assert lib.sf_status_string(4) == b"SF_ERR_WORKSPACE"
    assert lib.sf_status_string(99) == b"SF_ERR_UNKNOWN"
    assert lib.sf_version() >= 10000


def test_invalid_attention_shapes_are_rejected_on_the_host(lib):
    fake = ctypes.c_void_p(256)
    args = lambda B, n_q, H_q, H_kv, d, page: (fake, fake, fake, fake, fake, B, n_q, H_q, H_kv, d,
                                               page, 10, 4, 0.0, 0, fake, None, fake, 1 << 20,
                                               None)
    assert lib.sf_verify_attention(*args(0, 4, 8, 8, 64, 16)) == 1
    assert lib.sf_verify_attention(*args(1, 17, 8, 8, 64, 16)) == 1
    assert lib.sf_verify_attention(*args(1, 4, 7, 2, 64, 16)) == 1
    assert lib.sf_verify_attention(*args(1, 4, 8, 8, 96, 16)) == 2
    assert lib.sf_verify_attention(*args(1, 4, 8, 8, 64, 32)) == 2
    assert lib.sf_verify_attention(*args(1, 4, 32, 2, 64, 16)) == 2
    assert b"H_q" in lib.sf_last_error() or b"group" in lib.sf_last_error()
    assert lib.sf_verify_attention_workspace_size(0, 4, 8, 8, 64, 4, 16, 0) == 0
    null_q = list(args(1, 4, 8, 8, 64, 16))
    null_q[0] = None
    assert lib.sf_verify_attention(*null_q) == 1


def test_invalid_accept_arguments_are_rejected_on_the_host(lib):
    fake = ctypes.c_void_p(256)
    call = lambda B, k, V, ws=fake: lib.sf_accept(fake, fake, fake, fake, fake, B, k, V, fake,
                                                  fake, None, ws, 1 << 20, None)
    assert call(0, 4, 100) == 1
    assert call(2, 0, 100) == 1
    assert call(2, 17, 100) == 1
    assert call(2, 4, 1) == 1
    assert call(2, 4, 100, ws=None) == 4
    assert lib.sf_accept_workspace_size(2, 0, 100) == 0


def test_launch_counts_reject_invalid_shapes_before_touching_a_device():
    # shapes the calls would reject give 0 without any CUDA call
    lib = sfv.load_library()
    assert lib.sf_accept_kernel_launches(0, 5, 32000) == 0
    assert lib.sf_accept_kernel_launches(1, 17, 32000) == 0
    assert lib.sf_accept_kernel_launches(1, 5, 1) == 0
    assert lib.sf_verify_attention_kernel_launches(0, 5, 32, 32, 128, 189, 16, 0) == 0
    assert lib.sf_verify_attention_kernel_launches(1, 5, 32, 32, 96, 189, 16, 0) == 0
    assert lib.sf_verify_attention_kernel_launches(1, 5, 32, 32, 128, 189, 32, 0) == 0


def test_binding_rejects_host_tensors_and_bad_shapes_before_any_launch():
    # the binding checks dtype, device, contiguity and shapes before calling
    # the library; these run without a GPU because every check fails first
    import torch
    bf = torch.zeros((1, 4, 8, 64), dtype=torch.bfloat16)            # host tensor
    kc = torch.zeros((8, 8, 16, 64), dtype=torch.bfloat16)
    bt = torch.zeros((1, 8), dtype=torch.int32)
    sl = torch.full((1,), 20, dtype=torch.int32)
    with pytest.raises(ValueError, match="CUDA"):
        sfv.verify_attention(bf, kc, kc, bt, sl)
    with pytest.raises(TypeError, match="bfloat16"):
        sfv.verify_attention(bf.float(), kc, kc, bt, sl)
    with pytest.raises(ValueError, match="block_table"):
        sfv.verify_attention(bf, kc, kc, torch.zeros((2, 8), dtype=torch.int32), sl)
    with pytest.raises(ValueError, match="block_table"):
        sfv.verify_attention(bf, kc, kc, torch.zeros(8, dtype=torch.int32), sl)
    with pytest.raises(ValueError, match="CUDA"):
        sfv.read_device_status(torch.zeros(256, dtype=torch.uint8))
    with pytest.raises(TypeError, match="uint8"):
        sfv.workspace_init(torch.zeros(64, dtype=torch.int32))


def test_binding_rejects_a_cache_narrower_than_q_before_the_library_is_called(monkeypatch):
    # the library sizes the caches' tensor maps from q's head_dim, so a cache
    # with a smaller head_dim must be refused by the binding itself
    import torch

    def no_library():
        raise AssertionError("the library must not be reached")

    monkeypatch.setattr(sfv, "load_library", no_library)
    q = torch.zeros((1, 4, 8, 128), dtype=torch.bfloat16)
    kc = torch.zeros((8, 8, 16, 64), dtype=torch.bfloat16)
    bt = torch.zeros((1, 8), dtype=torch.int32)
    sl = torch.full((1,), 20, dtype=torch.int32)
    for fn in (sfv.verify_attention, sfv.verify_attention_noalloc):
        with pytest.raises(ValueError, match="head_dim"):
            fn(q, kc, kc, bt, sl)
