"""The permutation entry point that allocates nothing (moe_permute_noalloc)
against the workspace entry point (moe_permute), through the C ABI.

Some callers cannot give the library scratch memory (no device allocator of
their own, all memory reserved up front, or no cudaMalloc allowed where they
run); this entry point keeps its scratch in a static device array. Its
outputs must equal moe_permute's exactly, on two calls in a row (the second
call finds the first call's leftovers in the shared array)."""
import numpy as np
import pytest
import torch

import paper_2607_12875_gb300 as gb

pytestmark = pytest.mark.gpu


def _outputs(T, k, E):
    dev = "cuda"
    return (torch.empty(E, dtype=torch.int32, device=dev), torch.empty(E + 1, dtype=torch.int32, device=dev),
            torch.empty(T * k, dtype=torch.int32, device=dev), torch.empty(T * k, dtype=torch.int32, device=dev))


@pytest.mark.parametrize("T,k,E,seed", [(8192, 8, 128, 1), (333, 6, 64, 2)])
def test_noalloc_permute_equals_workspace_permute_twice(T, k, E, seed):
    cfg = gb.make_config(T, 4096, 1536, E, k, act="bf16", w="bf16")
    ws = torch.empty(gb.workspace_size(cfg), dtype=torch.uint8, device="cuda")
    gen = torch.Generator().manual_seed(seed)
    for call in range(2):
        ids = torch.randint(0, E, (T, k), generator=gen, dtype=torch.int32).cuda()
        ref = _outputs(T, k, E)
        got = _outputs(T, k, E)
        gb.moe_permute(cfg, ids, *ref, ws)
        gb.moe_permute_noalloc(cfg, ids, *got)
        torch.cuda.synchronize()
        for a, b in zip(ref, got):
            assert torch.equal(a, b), f"call {call}"
        assert int(ref[1][-1]) == T * k


def test_noalloc_permute_rejects_problems_beyond_its_scratch():
    # 2 * ceil(P/1024) * E ints must fit in 262144
    T, k, E = 65536, 8, 512
    cfg = gb.make_config(T, 4096, 1536, E, k, act="bf16", w="bf16")
    ids = torch.zeros((T, k), dtype=torch.int32, device="cuda")
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_permute_noalloc(cfg, ids, *_outputs(T, k, E))
    assert e.value.status == gb.EUNSUPPORTED
