"""Failure detection on the GPU without a GPU fault.

A bounded device wait that runs out is made to happen on purpose: an
internal entry point launches the fused product with every wait limited to
a few milliseconds and a grid barrier whose count is preset so that it never
opens.  Every CTA that holds records gives up at its final flush, sets the
handle's status word and returns; no kernel is left waiting.  The test then
checks that the timeout is reported on that handle only, that reading the
word clears it, and that the next call on the same handle is correct.

A kept list with an id out of range is the second planted failure
(DUO_EFORMAT): it is reported on the launch's handle, not on another one.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle as orc

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


def _case(O, I, seed):
    g = torch.Generator().manual_seed(seed)
    W = (torch.randn(O, I, generator=g) * 0.02).to(torch.float16)
    W[torch.rand(O, I, generator=g) < 0.5] = 0
    u = torch.rand(I, generator=g, dtype=torch.float64) - 0.5
    x = (-torch.sign(u) * torch.log1p(-2 * u.abs())).to(torch.float16)
    return W, x


def _check(y, W, x, k):
    Wn, xn = W.numpy(), x.numpy()
    K, _ = orc.oracle_sparsify(xn, k)
    err = np.abs(y.cpu().numpy().astype(np.float64) - orc.oracle_spmspv(Wn, xn, k))
    assert np.all(err <= orc.tolerance_rows(Wn, xn, K, 2e-3))


def test_wait_timeout_is_reported_and_the_handle_recovers(duo):
    lib = duo.load_library()
    O, I = 3000, 2048
    W, x = _case(O, I, 5)
    k = orc.k_from_pct(I, 50)
    h = duo.duo_pack(W.cuda(), "bitmask")
    other = duo.duo_pack(W.cuda(), "bitmask")
    xd = x.cuda()
    y = torch.empty(O, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    assert duo.duo_packed_status(h) == duo.DUO_OK
    rc = lib.duo_test_spmspv_blocked(h.handle, xd.data_ptr(), k, y.data_ptr(), 2_000_000, stream)
    assert rc == duo.DUO_OK   # the call returned: every wait gave up
    assert duo.duo_packed_status(other) == duo.DUO_OK   # not reported on another handle
    assert duo.duo_packed_status(h) == duo.DUO_ETIMEOUT
    assert duo.duo_packed_status(h) == duo.DUO_OK       # reading clears the word
    # the same handle, its own barrier: correct again
    for _ in range(2):
        y2 = duo.duo_spmspv(h, xd, k)
        torch.cuda.synchronize()
        _check(y2, W, x, k)
    assert duo.duo_packed_status(h) == duo.DUO_OK
    assert duo.duo_device_status() == duo.DUO_OK
    h.free()
    other.free()


def test_blocked_entry_rejects_long_limits(duo):
    lib = duo.load_library()
    W, x = _case(64, 64, 6)
    h = duo.duo_pack(W.cuda(), "bitmask")
    y = torch.empty(64, dtype=torch.float32, device="cuda")
    xd = x.cuda()
    stream = torch.cuda.current_stream().cuda_stream
    for limit in (0, 10**9):
        assert lib.duo_test_spmspv_blocked(h.handle, xd.data_ptr(), 32, y.data_ptr(), limit,
                                           stream) == duo.DUO_EINVAL
    h.free()


def test_bad_kept_id_is_reported_on_its_own_handle(duo):
    O, I = 2100, 777
    W, x = _case(O, I, 7)
    a = duo.duo_pack(W.cuda(), "bitmask")
    b = duo.duo_pack(W.cuda(), "bitmask")
    k = 40
    kidx = torch.arange(0, 2 * k, 2, dtype=torch.int16)   # uint16 ids, bit for bit
    kidx[7] = I + 5                      # out of range
    kval = x[: k].clone()
    duo.duo_spmspv(a, None, k, kept_idx=kidx.cuda(), kept_val=kval.cuda())
    torch.cuda.synchronize()
    assert duo.duo_packed_status(b) == duo.DUO_OK
    assert duo.duo_packed_status(a) == duo.DUO_EFORMAT
    # a's next call is correct
    y2 = duo.duo_spmspv(a, x.cuda(), k)
    torch.cuda.synchronize()
    _check(y2, W, x, k)
    assert duo.duo_packed_status(a) == duo.DUO_OK
    a.free()
    b.free()
