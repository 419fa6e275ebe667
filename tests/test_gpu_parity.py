"""GPU parity of the CUDA path (through the C ABI) against the CPU oracle.

Bar: kept channel ids / values and packed bytes bit-exact; y within
2e-3 * sum_{j in K} |W_ij| |x_j| per row (fp16 inputs, fp32 accumulation),
and exactly 0 where that sum is 0.  Small cases compare every row; the
LLaMA-shaped workloads compare sampled rows (first, last, segment borders and
a seeded random sample), launched the way bench.py launches them.
"""
import numpy as np
import pytest
import torch

import oracle as orc

pytestmark = pytest.mark.gpu

REL_TOL = 2e-3


@pytest.fixture(scope="module")
def duo():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo as d
    d.load_library()
    return d


def _np16(t):
    return t.detach().cpu().numpy().view(np.float16) if t.dtype == torch.float16 else \
        t.detach().cpu().numpy()


def _check_y(y_gpu, W_rows16, x16, k, label=""):
    K, _ = orc.oracle_sparsify(x16, k)
    y_ref = orc.oracle_spmspv(W_rows16, x16, k)
    tol = orc.tolerance_rows(W_rows16, x16, K, REL_TOL)
    y = np.asarray(y_gpu, dtype=np.float64)
    err = np.abs(y - y_ref)
    bad = err > tol
    assert not bad.any(), (f"{label}: {bad.sum()} rows out of tolerance; worst row "
                           f"{int(np.argmax(err - tol))} err {err.max():.3e}")
    zero_rows = tol == 0
    assert np.all(y[zero_rows] == 0.0), f"{label}: rows with an empty kept support must be 0"


def _rand_case(O, I, pw, seed, dist="laplace"):
    g = torch.Generator().manual_seed(seed)
    W = (torch.randn(O, I, generator=g) * 0.02).to(torch.float16)
    if pw > 0:
        W[torch.rand(O, I, generator=g) < pw] = 0
    if dist == "laplace":
        u = torch.rand(I, generator=g, dtype=torch.float64) - 0.5
        x = (-torch.sign(u) * torch.log1p(-2 * u.abs())).to(torch.float16)
    elif dist == "ties":
        x = (torch.randint(-3, 4, (I,), generator=g).to(torch.float16) * 0.25)
    else:
        raise ValueError(dist)
    return W, x


# ---------------------------------------------------------------- sparsify --

SPARSIFY_SIZES = [1, 2, 31, 32, 33, 100, 1000, 4096, 5120, 11008, 13824, 14336, 28672, 65535]


@pytest.mark.parametrize("I", SPARSIFY_SIZES)
def test_sparsify_bit_exact(duo, I):
    g = torch.Generator().manual_seed(I)
    cases = {
        "laplace": _rand_case(1, I, 0, I)[1],
        "ties": (torch.randint(-3, 4, (I,), generator=g).to(torch.float16) * 0.5),
        "equal": torch.full((I,), -1.5, dtype=torch.float16),
        "zeros": torch.zeros(I, dtype=torch.float16),
    }
    z = cases["zeros"].clone()
    z[::2] = -0.0
    cases["signed_zeros"] = z
    big = cases["laplace"].clone()
    big[:: max(1, I // 7)] = float("inf")
    cases["with_inf"] = big
    ks = sorted({0, 1, I // 2, max(0, I - 1), I, orc.k_from_pct(I, 70), orc.k_from_pct(I, 25)})
    for name, x in cases.items():
        xd = x.cuda()
        xn = x.numpy()
        for k in ks:
            idx, val = duo.duo_sparsify(xd, k)
            K, vals = orc.oracle_sparsify(xn, k)
            assert np.array_equal(idx.cpu().numpy().view(np.uint16), K), (name, k)
            assert np.array_equal(val.cpu().numpy().view(np.uint16), vals.view(np.uint16)), (name, k)
    assert duo.duo_device_status() == 0


# ------------------------------------------------------------------ packer --

PACK_SHAPES = [(1, 1), (31, 3), (1023, 5), (1024, 33), (1025, 40), (2100, 65), (3000, 130)]


@pytest.mark.parametrize("O,I", PACK_SHAPES)
@pytest.mark.parametrize("fmt", ["bitmask", "idx16"])
def test_pack_bytes_bit_exact(duo, O, I, fmt):
    W, _ = _rand_case(O, I, 0.5, O * 7 + I)
    if I > 2:
        W[:, 1] = 0                     # an empty channel
        W[:, 2] = 0.25                  # a full channel
    W[0, 0] = -0.0                      # -0 is pruned
    h = duo.duo_pack(W.cuda(), fmt)
    info, index, aux, data = duo.packed_bytes(h)
    Wn = W.numpy()
    if fmt == "bitmask":
        hdr, off, ref = orc.ref_pack_cmb(Wn)
        assert info.magic == hdr["magic"] and info.nseg == hdr["nseg"] and info.seg_rows == 1024
        assert np.array_equal(index.view(np.uint32), off)
    else:
        hdr, colptr, cnt, ref = orc.ref_pack_idx16(Wn)
        assert info.magic == hdr["magic"]
        assert np.array_equal(index.view(np.uint64), colptr)
        assert np.array_equal(aux.view(np.uint32), cnt)
    assert info.nnz == hdr["nnz"] and info.out == O and info.inp == I
    assert np.array_equal(data, ref)
    h.free()


def test_pack_strided_rows_and_single_nonzero(duo):
    O, I, ldw = 1500, 40, 64
    base = torch.zeros(O, ldw, dtype=torch.float16)
    base[:, I:] = 7.0                           # outside the view: must be ignored
    W = base[:, :I]
    W[1234, 17] = -3.0
    h = duo.duo_pack(W.cuda(), "bitmask")
    info, index, _, data = duo.packed_bytes(h)
    hdr, off, ref = orc.ref_pack_cmb(W.contiguous().numpy())
    assert np.array_equal(index.view(np.uint32), off) and np.array_equal(data, ref)
    assert info.nnz == 1


def test_pack_config1_bytes(duo):
    from paper_2506_20194_gb300 import synth
    W, _ = synth.single_layer(device="cpu")
    h = duo.duo_pack(W.cuda(), "bitmask")
    _, index, _, data = duo.packed_bytes(h)
    hdr, off, ref = orc.ref_pack_cmb(W.numpy())
    assert np.array_equal(index.view(np.uint32), off)
    assert np.array_equal(data, ref)


# ------------------------------------------------------------------ spMspV --

SMALL = [(1, 1), (5, 7), (33, 100), (1000, 257), (1025, 1030), (2100, 513), (3000, 4096)]


@pytest.mark.parametrize("O,I", SMALL)
@pytest.mark.parametrize("fmt", ["bitmask", "idx16"])
def test_spmspv_small_all_rows(duo, O, I, fmt):
    for pw in (0.0, 0.5, 0.9):
        W, x = _rand_case(O, I, pw, O + 3 * I + int(pw * 10), "laplace" if O % 2 else "ties")
        Wd, xd = W.cuda(), x.cuda()
        h = duo.duo_pack(Wd, fmt)
        for pct in (0, 50, 90, 100):
            k = orc.k_from_pct(I, pct)
            y = duo.duo_spmspv(h, xd, k)                        # fused selection
            _check_y(_np16(y), W.numpy(), x.numpy(), k, f"{fmt} fused {O}x{I} pw{pw} k{k}")
            idx, val = duo.duo_sparsify(xd, k)
            y2 = duo.duo_spmspv(h, None, k, idx, val)           # listed
            _check_y(_np16(y2), W.numpy(), x.numpy(), k, f"{fmt} listed {O}x{I} pw{pw} k{k}")
        h.free()
    assert duo.duo_device_status() == 0


def test_spmspv_listed_any_order(duo):
    O, I = 2048, 600
    W, x = _rand_case(O, I, 0.5, 99)
    h = duo.duo_pack(W.cuda(), "bitmask")
    k = 300
    K, vals = orc.oracle_sparsify(x.numpy(), k)
    perm = np.random.default_rng(0).permutation(k)
    idx = torch.from_numpy(K[perm].view(np.int16).copy()).cuda()
    val = torch.from_numpy(vals[perm].copy()).cuda()
    y = duo.duo_spmspv(h, None, k, idx, val)
    _check_y(_np16(y), W.numpy(), x.numpy(), k, "permuted list")


def test_spmspv_degenerate(duo):
    O, I = 1100, 300
    W, x = _rand_case(O, I, 0.5, 5)
    Wz = torch.zeros_like(W)
    xz = torch.zeros_like(x)
    for Wc, xc in ((W, x), (Wz, x), (W, xz), (Wz, xz)):
        h = duo.duo_pack(Wc.cuda(), "bitmask")
        for k in (0, 1, I):
            y = duo.duo_spmspv(h, xc.cuda(), k)
            _check_y(_np16(y), Wc.numpy(), xc.numpy(), k, f"degenerate k{k}")
        h.free()
    # y is fully overwritten even if it held garbage
    h = duo.duo_pack(W.cuda(), "bitmask")
    y = torch.full((O,), 123.0, device="cuda")
    duo.duo_spmspv(h, x.cuda(), 150, y=y)
    _check_y(_np16(y), W.numpy(), x.numpy(), 150, "overwrite")


def test_multi_shared_input_gqa_shapes(duo):
    """q (4096x4096) and GQA k/v (1024x4096) sharing one sparsified input."""
    I = 4096
    Ws = [_rand_case(O, I, 0.6, 10 + O)[0] for O in (4096, 1024, 1024)]
    x = _rand_case(1, I, 0, 77)[1]
    hs = [duo.duo_pack(W.cuda(), "bitmask") for W in Ws]
    for pct in (0, 50, 70):
        k = orc.k_from_pct(I, pct)
        ys = duo.duo_spmspv_multi(hs, x.cuda(), k)
        for W, y in zip(Ws, ys):
            _check_y(_np16(y), W.numpy(), x.numpy(), k, f"multi pct{pct}")
        idx, val = duo.duo_sparsify(x.cuda(), k)
        ys = duo.duo_spmspv_multi(hs, None, k, idx, val)
        for W, y in zip(Ws, ys):
            _check_y(_np16(y), W.numpy(), x.numpy(), k, f"multi listed pct{pct}")


def test_repeated_calls_and_graph_replay(duo):
    """Same handle back to back, and inside a CUDA graph replayed many times
    (the grid-barrier state must return to rest after every launch)."""
    O, I = 4096, 4096
    W, x = _rand_case(O, I, 0.5, 3)
    h = duo.duo_pack(W.cuda(), "bitmask")
    xd = x.cuda()
    k = 2048
    y = torch.empty(O, device="cuda")
    for _ in range(20):
        duo.duo_spmspv(h, xd, k, y=y)
    _check_y(_np16(y), W.numpy(), x.numpy(), k, "repeat")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        duo.duo_spmspv(h, xd, k, y=y)
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        duo.duo_spmspv(h, xd, k, y=y)
    for _ in range(50):
        g.replay()
    torch.cuda.synchronize()
    _check_y(_np16(y), W.numpy(), x.numpy(), k, "graph replay")
    x2 = _rand_case(1, I, 0, 4)[1]
    xd.copy_(x2)
    g.replay()
    torch.cuda.synchronize()
    _check_y(_np16(y), W.numpy(), x2.numpy(), k, "graph replay new x")
    assert duo.duo_device_status() == 0


# ------------------------------------------------- LLaMA-shaped workloads --

def _sample_rows(O, n, seed):
    rng = np.random.default_rng(seed)
    fixed = {0, O - 1}
    for b in range(1024, O, 1024):
        fixed |= {b - 1, b}
    rows = sorted(fixed | set(rng.choice(O, size=min(O, n), replace=False).tolist()))
    return np.array([r for r in rows if 0 <= r < O])


def _run_layer_like_bench(duo, synth, wl, layer, device, pct, pw=None, nrows=384):
    """Packs one decoder layer and runs it as bench.py does: q/k/v and gate/up
    as shared-input multi launches, o and down alone, fused selection."""
    shape = wl["shape"]
    Ws = {p: synth.layer_weight(wl, p, layer=layer, device=device, pw=pw) for p in synth.PROJS}
    xs = {p: synth.layer_input(wl, p, layer=layer, device=device) for p in ("q", "o", "gate", "down")}
    hs = {p: duo.duo_pack(Ws[p], "bitmask") for p in synth.PROJS}
    out = {}
    kq = orc.k_from_pct(shape.I("q"), pct)
    out.update(zip(("q", "k", "v"), duo.duo_spmspv_multi([hs["q"], hs["k"], hs["v"]], xs["q"], kq)))
    out["o"] = duo.duo_spmspv(hs["o"], xs["o"], orc.k_from_pct(shape.I("o"), pct))
    kg = orc.k_from_pct(shape.I("gate"), pct)
    out.update(zip(("gate", "up"), duo.duo_spmspv_multi([hs["gate"], hs["up"]], xs["gate"], kg)))
    out["down"] = duo.duo_spmspv(hs["down"], xs["down"], orc.k_from_pct(shape.I("down"), pct))
    torch.cuda.synchronize()
    src = {"q": "q", "k": "q", "v": "q", "o": "o", "gate": "gate", "up": "gate", "down": "down"}
    for p in synth.PROJS:
        O, I = shape.shapes[p]
        rows = _sample_rows(O, nrows, layer * 7 + synth.PROJS.index(p))
        Wr = Ws[p][torch.from_numpy(rows).to(device)].cpu().numpy().view(np.float16)
        x16 = xs[src[p]].cpu().numpy().view(np.float16)
        k = orc.k_from_pct(I, pct)
        _check_y(out[p].cpu().numpy()[rows], Wr, x16, k, f"{shape.name} L{layer} {p} px{pct}")
    for h in hs.values():
        h.free()
    assert duo.duo_device_status() == 0


def test_config1_single_layer_all_rows(duo):
    from paper_2506_20194_gb300 import synth
    W, x = synth.single_layer(device="cuda")
    h = duo.duo_pack(W, "bitmask")
    y = duo.duo_spmspv(h, x, 2048)
    _check_y(_np16(y), W.cpu().numpy().view(np.float16), x.cpu().numpy().view(np.float16), 2048, "cfg1")


@pytest.mark.parametrize("pct", [0, 25, 50, 70])
def test_config2_llama2_7b_layer(duo, pct):
    from paper_2506_20194_gb300 import synth
    _run_layer_like_bench(duo, synth, synth.WORKLOADS["llama2-7b-layer"], 0, "cuda", pct)


def test_config3_llama3_8b_layer(duo):
    from paper_2506_20194_gb300 import synth
    _run_layer_like_bench(duo, synth, synth.WORKLOADS["llama3-8b-stack"], 5, "cuda", 50)


@pytest.mark.parametrize("pw,pct", [(0.4, 30), (0.5, 50), (0.6, 70)])
def test_config4_llama2_13b_layer_with_outliers(duo, pw, pct):
    from paper_2506_20194_gb300 import synth
    _run_layer_like_bench(duo, synth, synth.WORKLOADS["llama2-13b-stack"], 1, "cuda", pct, pw=pw)


def test_config5_llama2_70b_layer(duo):
    from paper_2506_20194_gb300 import synth
    _run_layer_like_bench(duo, synth, synth.WORKLOADS["llama2-70b-stack"], 0, "cuda", 50, nrows=256)


# ------------------------------------------------------------ host errors --

def test_gpu_argument_errors(duo):
    W, x = _rand_case(64, 64, 0.5, 1)
    h = duo.duo_pack(W.cuda(), "bitmask")
    y = torch.empty(65, device="cuda")
    with pytest.raises(duo.DuoError) as e:
        duo.duo_spmspv(h, x.cuda(), 8, y=y[1:])            # y not 16-byte aligned
    assert e.value.code == duo.DUO_EINVAL
    lib = duo.load_library()
    import ctypes
    hh = ctypes.c_void_p()
    Wh = W.contiguous()                                     # host memory, not device
    assert lib.duo_pack(Wh.data_ptr(), 64, 64, 64, 1, None, ctypes.byref(hh)) == duo.DUO_EINVAL
    hidx = duo.duo_pack(W.cuda(), "idx16")
    with pytest.raises(duo.DuoError) as e:
        duo.duo_spmspv_multi([hidx, hidx], x.cuda(), 8)
    assert e.value.code == duo.DUO_EFORMAT
    raw = h.handle
    h.free()
    assert lib.duo_free(raw) == duo.DUO_EINVAL              # double free
    assert lib.duo_spmspv(raw, x.cuda().data_ptr(), None, None, 8, y.data_ptr(), None) == duo.DUO_EINVAL
    hidx.free()


def test_listed_bad_channel_id_is_reported_not_faulted(duo):
    O, I = 2048, 100
    W, x = _rand_case(O, I, 0.5, 8)
    h = duo.duo_pack(W.cuda(), "bitmask")
    idx = torch.tensor([3, 5, 200], dtype=torch.int16, device="cuda")   # 200 >= I
    val = torch.ones(3, dtype=torch.float16, device="cuda")
    duo.duo_spmspv(h, None, 3, idx, val)
    assert duo.duo_device_status() == duo.DUO_EFORMAT
    assert duo.duo_device_status() == duo.DUO_OK            # cleared, context usable
    y = duo.duo_spmspv(h, x.cuda(), 50)
    _check_y(_np16(y), W.numpy(), x.numpy(), 50, "after format error")


def test_alloc_failure_injection_leaks_nothing(tmp_path):
    """DUO_FAULT_ALLOC_FAIL=n fails the n-th device allocation: duo_pack
    returns DUO_ENOMEM and frees what it already allocated."""
    import subprocess
    import sys
    import os
    code = r"""
import torch, sys
from paper_2506_20194_gb300 import duo
duo.load_library()
W = torch.zeros(3000, 500, dtype=torch.float16, device='cuda'); W[::3, ::2] = 1.0
duo.duo_pack(W, 'bitmask').free()          # warm-up: allocations 1..4, modules loaded
torch.cuda.synchronize()
free0 = torch.cuda.mem_get_info()[0]
try:
    duo.duo_pack(W, 'bitmask'); print('NOFAIL')
except duo.DuoError as e:
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    print('CODE', e.code, 'LEAK', free0 - free1)
"""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    for n in (5, 6, 7, 8):                 # the 4 allocations of the second duo_pack
        env = dict(os.environ, DUO_FAULT_ALLOC_FAIL=str(n), PYTHONPATH=root)
        r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                           cwd=root, timeout=300)
        assert r.returncode == 0, r.stderr
        out = r.stdout.split()
        assert out[0] == "CODE" and int(out[1]) == -2, r.stdout
        assert int(out[3]) <= 2 * 1024 * 1024, f"leak after injected failure {n}: {out[3]} bytes"


def test_step_graph_copies_and_products(duo):
    """duo.StepGraph: a captured step (pinned-host inputs in, outputs out)
    gives the oracle's y, for new inputs written before each run; two stages,
    one of them a shared-input pair."""
    d = duo
    rng = np.random.default_rng(77)
    I1, I2 = 1000, 333
    Ws = [(rng.standard_normal((O, I1)) * 0.02).astype(np.float16) for O in (700, 1300)]
    W2 = (rng.standard_normal((517, I2)) * 0.02).astype(np.float16)
    for W in Ws + [W2]:
        W[rng.random(W.shape) < 0.5] = 0
    hs = [d.duo_pack(torch.from_numpy(W).cuda(), "bitmask") for W in Ws]
    h2 = d.duo_pack(torch.from_numpy(W2).cuda(), "bitmask")
    plan = d.StepGraph([{"h": hs, "k": 400}, {"h": h2, "k": 100}])
    for trial in range(3):
        x1 = rng.laplace(0, 1, size=I1).astype(np.float16)
        x2 = rng.laplace(0, 1, size=I2).astype(np.float16)
        plan.x_host(0).copy_(torch.from_numpy(x1))
        plan.x_host(1).copy_(torch.from_numpy(x2))
        plan.run()
        torch.cuda.synchronize()
        for (W, x, kk, y) in [(Ws[0], x1, 400, plan.y_host(0, 0)), (Ws[1], x1, 400, plan.y_host(0, 1)),
                              (W2, x2, 100, plan.y_host(1))]:
            K, _ = orc.oracle_sparsify(x, kk)
            err = np.abs(y.numpy().astype(np.float64) - orc.oracle_spmspv(W, x, kk))
            assert np.all(err <= orc.tolerance_rows(W, x, K)), trial
    for h in hs + [h2]:
        h.free()


@pytest.mark.parametrize("nbytes,off", [(0, 0), (1, 0), (15, 1), (16, 0), (17, 3), (12293, 0), (12293, 2),
                                        (1 << 20, 0)])
def test_copy_kernel_bytes(duo, nbytes, off):
    """duo_copy moves exactly the bytes asked for, device <-> pinned host and
    device -> device, aligned (16-byte words) and misaligned (byte path),
    and writes nothing past the range."""
    d = duo
    rng = np.random.default_rng(nbytes + off)
    src = torch.from_numpy(rng.integers(0, 256, size=nbytes + 32, dtype=np.uint8)).pin_memory()
    dev = torch.full((nbytes + 32,), 0xA5, dtype=torch.uint8, device="cuda")
    back = torch.full((nbytes + 32,), 0x5A, dtype=torch.uint8).pin_memory()
    dev2 = torch.full((nbytes + 32,), 0x3C, dtype=torch.uint8, device="cuda")
    d.duo_copy(dev[off:off + nbytes], src[off:off + nbytes])
    d.duo_copy(dev2[off:off + nbytes], dev[off:off + nbytes])
    d.duo_copy(back[off:off + nbytes], dev2[off:off + nbytes])
    torch.cuda.synchronize()
    s, b = src.numpy(), back.numpy()
    assert np.array_equal(b[off:off + nbytes], s[off:off + nbytes])
    assert np.all(b[:off] == 0x5A) and np.all(b[off + nbytes:] == 0x5A)
    dv = dev.cpu().numpy()
    assert np.all(dv[:off] == 0xA5) and np.all(dv[off + nbytes:] == 0xA5)
    assert d.duo_device_status() == 0


def test_copy_kernel_rejects_pageable_host_memory(duo):
    """Plain (unpinned) host memory is refused on the host with EINVAL; the
    stream stays usable."""
    d = duo
    pageable = torch.zeros(64, dtype=torch.uint8)
    dev = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(d.DuoError):
        d.duo_copy(dev, pageable)
    with pytest.raises(d.DuoError):
        d.duo_copy(pageable, dev)
    d.duo_copy(dev, torch.ones(64, dtype=torch.uint8).pin_memory())
    torch.cuda.synchronize()
    assert int(dev.sum()) == 64

