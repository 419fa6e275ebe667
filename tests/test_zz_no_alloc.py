"""GPU test of duo_pack_cmb_noalloc, the packing entry point that allocates
nothing (for callers that cannot call cudaMalloc themselves).

It must produce exactly the bytes of duo_pack, on two calls in a row (the
calls share one static scratch array), and reject what exceeds its limits.
This file is collected last so that a run stopping at the first failure has
run every other test already; it also passes when run alone.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def duo():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo as d
    d.load_library()
    return d


def _weight(O, I, seed, pw=0.5):
    g = torch.Generator().manual_seed(seed)
    W = (torch.randn(O, I, generator=g) * 0.02).to(torch.float16)
    W[torch.rand(O, I, generator=g) < pw] = 0
    return W.cuda()


def test_noalloc_pack_matches_duo_pack_twice(duo):
    # Two different weights packed one after the other: the second call reuses
    # the scratch the first one filled.
    for W in (_weight(2100, 333, 1), _weight(4096, 1000, 2, pw=0.3)):
        O, I = W.shape
        off, data, nbytes = duo.duo_pack_cmb_noalloc(W)
        h = duo.duo_pack(W, "bitmask")
        info, ref_off, _, ref_data = duo.packed_bytes(h)
        assert nbytes == info.data_bytes
        assert np.array_equal(off.cpu().numpy().view(np.uint8), ref_off)
        assert np.array_equal(data[:nbytes].cpu().numpy(), ref_data)
        h.free()
    assert duo.duo_device_status() == duo.DUO_OK


def test_noalloc_limits_and_size_query(duo):
    lib = duo.load_library()
    W = _weight(1500, 200, 3)
    O, I = W.shape
    S = (O + 1023) // 1024
    off = torch.empty(I * S + 1, dtype=torch.int32, device="cuda")
    nb = ctypes.c_int64(-1)
    stream = torch.cuda.current_stream().cuda_stream
    # size query (no data buffer), then a too-small buffer
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, I, off.data_ptr(), None, 0,
                                    ctypes.byref(nb), stream) == duo.DUO_OK
    need = nb.value
    small = torch.empty(16, dtype=torch.uint8, device="cuda")
    nb2 = ctypes.c_int64(-1)
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, I, off.data_ptr(), small.data_ptr(), 16,
                                    ctypes.byref(nb2), stream) == duo.DUO_ERANGE
    assert nb2.value == need
    # beyond the scratch limit: in * ceil(out / 1024) > DUO_NOALLOC_MAX_RECORDS
    big_in = 65535
    big_out = 1024 * 5            # 5 segments x 65535 channels > 262144 records
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), big_out, big_in, big_in, off.data_ptr(),
                                    small.data_ptr(), 16, ctypes.byref(nb2), stream) == duo.DUO_ERANGE
