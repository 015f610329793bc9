"""The allocation-free selection entry point against the allocating one.

lazymar_select_tokens_noalloc exists for callers that may not allocate device
memory once they are running: a serving loop that fixes its memory budget at
start-up, or a plug-in whose host framework owns the device allocator. Its
similarity scratch is a fixed array inside the library instead of
stream-ordered allocations.

This file is collected last so that a run stopping at the first failure has
already run every other test. It calls the new entry point twice in a row
through the C ABI, each time on a copy of the inputs given to
lazymar_select_tokens, and requires the same results with the tolerance every
selection test uses: identical indices, bit for bit, and an identical updated
reference tensor.
"""
import pytest

import synth
from paper_2503_12450_gb300 import lazymar as lm
from _gpu import DT, dev, sync, torch_cuda

pytestmark = pytest.mark.gpu

# Two calls in a row with different shapes: the second finds the first call's
# similarities still in the shared scratch.
CASES = [(64, 320, 768, 50, "bf16", 901), (32, 1088, 1024, 272, "bf16", 902)]


def test_noalloc_selection_matches_allocating_entry_point_on_two_calls():
    torch = torch_cuda()
    for rows, T, D, N, dtype, seed in CASES:
        cur, ref = synth.similarity_inputs(rows, T, D, seed=seed, dtype=dtype)
        a_cur, a_ref = dev(cur, dtype), dev(ref, dtype)
        b_cur, b_ref = dev(cur, dtype), dev(ref, dtype)
        idx_a = torch.full((rows, N), -1, dtype=torch.int32, device="cuda")
        idx_b = torch.full((rows, N), -2, dtype=torch.int32, device="cuda")
        lm.lazymar_select_tokens(DT[dtype], a_cur, a_ref, rows, T, D, N, idx_a)
        lm.lazymar_select_tokens_noalloc(DT[dtype], b_cur, b_ref, rows, T, D, N, idx_b)
        sync()
        assert torch.equal(idx_a, idx_b)
        assert torch.equal(a_ref, b_ref) and torch.equal(b_ref, b_cur)


# fp32 inputs; no token recomputed; T = 8192, where the top-N's key array
# (64 KiB) needs the opt-in shared-memory size; rows x T at the limit.
MORE_CASES = [(2, 80, 256, 20, "fp32", 903), (3, 320, 768, 0, "bf16", 904), (16, 8192, 64, 1000, "bf16", 905),
              (256, 1024, 8, 100, "bf16", 906)]


@pytest.mark.parametrize("rows,T,D,N,dtype,seed", MORE_CASES)
def test_noalloc_selection_more_shapes(rows, T, D, N, dtype, seed):
    torch = torch_cuda()
    cur, ref = synth.similarity_inputs(rows, T, D, seed=seed, dtype=dtype)
    a_cur, a_ref = dev(cur, dtype), dev(ref, dtype)
    b_cur, b_ref = dev(cur, dtype), dev(ref, dtype)
    idx_a = torch.full((rows, max(N, 1)), -1, dtype=torch.int32, device="cuda")
    idx_b = torch.full((rows, max(N, 1)), -2, dtype=torch.int32, device="cuda")
    lm.lazymar_select_tokens(DT[dtype], a_cur, a_ref, rows, T, D, N, idx_a)
    lm.lazymar_select_tokens_noalloc(DT[dtype], b_cur, b_ref, rows, T, D, N, idx_b)
    sync()
    assert torch.equal(idx_a[:, :N], idx_b[:, :N])
    assert torch.equal(a_ref, b_ref) and torch.equal(b_ref, b_cur)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    torch_cuda()
    # 257 rows x 1024 tokens = 263,168 > LAZYMAR_SELECT_NOALLOC_MAX_TOKENS (262,144);
    # refused before any device work.
    with pytest.raises(lm.LazymarError) as e:
        lm.lazymar_select_tokens_noalloc(lm.LAZYMAR_BF16, 0, 0, 257, 1024, 8, 1, 0)
    assert e.value.status == 1
    assert "LAZYMAR_SELECT_NOALLOC_MAX_TOKENS" in str(e.value)
