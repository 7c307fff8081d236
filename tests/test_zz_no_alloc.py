"""sf_verify_attention_noalloc against sf_verify_attention (GPU, C ABI).

The no-allocation entry point serves callers that cannot allocate device
memory while they verify (a serving runtime that owns all device memory, a
plug-in handed only its buffers); it runs the same kernel on the library's
own device scratch.  Two calls in a row, on different shapes, must each match
the workspace entry point within the parity tolerances of the other tests,
so no state left in the shared scratch leaks into the next call.  This file
is collected last on purpose.
"""
import numpy as np
import pytest
import torch

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import make_attention_case
from tests.gpu_helpers import (ATTN_LSE_ATOL, ATTN_OUT_ATOL, attention_to_device, require_gpu)

pytestmark = pytest.mark.gpu


def test_noalloc_matches_the_workspace_entry_point_on_two_calls():
    require_gpu()
    cases = [make_attention_case(4, 8, 28, 4, 128, [4864, 1200, 3600, 63], seed=501),
             make_attention_case(2, 5, 32, 32, 128, [3008, 17], seed=502)]
    for case in cases:
        dev = attention_to_device(case)
        args = (dev["q"], dev["k_cache"], dev["v_cache"], dev["block_table"], dev["seq_lens"])
        ref_out, ref_lse = sfv.verify_attention(*args)
        out, lse = sfv.verify_attention_noalloc(*args)
        torch.cuda.synchronize()
        err_o = (out.float() - ref_out.float()).abs().max().item()
        err_l = (lse - ref_lse).abs().max().item()
        assert np.isfinite(err_o) and np.isfinite(err_l)
        assert err_o <= ATTN_OUT_ATOL and err_l <= ATTN_LSE_ATOL, (err_o, err_l)
