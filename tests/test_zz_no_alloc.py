"""sf_verify_attention_noalloc against sf_verify_attention (GPU, C ABI).

The no-allocation entry point serves callers that cannot allocate device
memory while they verify (a serving runtime that owns all device memory, a
plug-in handed only its buffers); it runs the same kernels, with the same
launch plan, on the library's own device scratch.  Its results must therefore
equal the workspace entry point's bit for bit.  The calls run in a row,
smaller shape first, so the larger call finds the smaller one's descriptors,
tickets and partials in the shared scratch: any of that state leaking into the
next call would show as a difference.  A shape whose workspace exceeds the
built-in scratch must be refused before anything is enqueued.  This file is
collected last on purpose.
"""
import pytest
import torch

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import make_attention_case
from tests.gpu_helpers import attention_to_device, require_gpu

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 16 << 20  # the built-in scratch of sf_verify_attention_noalloc


def test_noalloc_equals_the_workspace_entry_point_on_calls_in_a_row():
    require_gpu()
    cases = [make_attention_case(2, 5, 32, 32, 128, [3008, 17], seed=502),       # mma.sync kernel
             make_attention_case(4, 8, 28, 4, 128, [4864, 1200, 3600, 63], seed=501),  # tcgen05
             make_attention_case(1, 6, 28, 4, 128, [2000], seed=503)]
    for case in cases:
        dev = attention_to_device(case)
        args = (dev["q"], dev["k_cache"], dev["v_cache"], dev["block_table"], dev["seq_lens"])
        ref_out, ref_lse = sfv.verify_attention(*args)
        out, lse = sfv.verify_attention_noalloc(*args)
        torch.cuda.synchronize()
        assert torch.equal(out, ref_out)
        assert torch.equal(lse, ref_lse)


def test_noalloc_refuses_a_shape_beyond_its_scratch():
    require_gpu()
    B, n_q, H_q, H_kv, d = 64, 16, 32, 4, 128
    need = sfv.verify_attention_workspace_size(B, n_q, H_q, H_kv, d, 1)
    assert need > SCRATCH_BYTES
    q = torch.zeros((B, n_q, H_q, d), dtype=torch.bfloat16, device="cuda")
    kc = torch.zeros((B, H_kv, 16, d), dtype=torch.bfloat16, device="cuda")
    bt = torch.arange(B, dtype=torch.int32, device="cuda").view(B, 1)
    sl = torch.full((B,), n_q, dtype=torch.int32, device="cuda")
    out = torch.full_like(q, 7.0)
    with pytest.raises(sfv.SFError) as err:
        sfv.verify_attention_noalloc(q, kc, kc, bt, sl, out=out)
    assert err.value.status == 2  # SF_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())  # nothing was launched
