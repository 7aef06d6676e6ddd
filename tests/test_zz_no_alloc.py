"""The slot check that allocates nothing, against the one that takes caller scratch.

`stepq_validate_slots_noalloc` serves callers that cannot allocate device memory
and have no scratch buffer of their own to pass (for example code running where
a host framework owns every device allocation): it keeps its bitmap in a fixed
device array inside the library. Its answers must equal those of
`stepq_validate_slots` on the same slot lists, call after call. This file sorts
last so that a stop-at-first-failure run has already run every other test.
"""
import ctypes as C

import pytest

pytestmark = pytest.mark.gpu


def test_noalloc_slot_check_matches_scratch_version():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_38169_gb300 import _lib
    L = _lib.lib()
    dev = torch.device("cuda", 0)
    stream = C.c_void_p(torch.cuda.current_stream(dev).cuda_stream)
    pool_slots = 5000
    scratch = torch.zeros((pool_slots + 31) // 32, dtype=torch.int32, device=dev)
    cases = [
        [3, 17, 4999, 0, 1024],          # distinct and in range
        [7, 9, 7],                       # a repeat
        [12, 5000],                      # out of range
        list(range(0, 5000, 3)),         # many distinct
        [4999, 4999],                    # a repeat at the top bit of the last word
    ]
    expected = [0, 3, 2, 0, 3]           # STEPQ_OK, _DUP_SLOT, _SLOT_RANGE, _OK, _DUP_SLOT
    for _round in range(2):              # two calls in a row per case, then all again
        for case, want in zip(cases, expected):
            slots = torch.tensor(case, dtype=torch.int32, device=dev)
            ref = torch.full((1,), -1, dtype=torch.int32, device=dev)
            got = torch.full((1,), -1, dtype=torch.int32, device=dev)
            assert L.stepq_validate_slots(C.c_void_p(slots.data_ptr()), len(case), pool_slots,
                                          C.c_void_p(scratch.data_ptr()), C.c_void_p(ref.data_ptr()),
                                          stream) == 0
            for _ in range(2):
                got.fill_(-1)
                assert L.stepq_validate_slots_noalloc(C.c_void_p(slots.data_ptr()), len(case),
                                                      pool_slots, C.c_void_p(got.data_ptr()),
                                                      stream) == 0
                torch.cuda.synchronize(dev)
                assert int(got.item()) == int(ref.item()) == want, (case, int(got.item()), int(ref.item()))
    # a pool beyond the fixed array is refused before any work
    one = torch.zeros(1, dtype=torch.int32, device=dev)
    assert L.stepq_validate_slots_noalloc(C.c_void_p(one.data_ptr()), 1, (1 << 20) + 1,
                                          C.c_void_p(one.data_ptr()), stream) == 7
    assert L.stepq_device_error(stream) == 0
