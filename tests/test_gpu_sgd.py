"""The model update after the aggregation (Eq. 1 with heavy-ball momentum):
aspis_sgd against the oracle, bit for bit, on seeded inputs of several
lengths (ragged tails), both load paths, with and without momentum, aliased
arrays, IEEE special values, the full ResNet-18 gradient length, and chained
after the round on the round's own output.  Argument errors are checked
without a GPU."""
import ctypes
import dataclasses

import numpy as np
import pytest

import oracle
import synth

ap = pytest.importorskip("paper_2108_02416_gb300")


# ------------------------------------------------------------- no GPU needed

def _call(g, w, v, d, eta=0.1, mu=0.9):
    P = ctypes.c_void_p
    return ap.lib.aspis_sgd(P(g), P(w), P(v), d, eta, mu, None)


def test_sgd_rejects_bad_arguments():
    # returned before anything reaches the device: fake, never dereferenced addresses
    g, w, v = 0x10000, 0x20000, 0x30000
    assert _call(g, w, v, -1) == ap.E_INVAL
    assert _call(None, w, v, 8) == ap.E_INVAL
    assert _call(g, None, v, 8) == ap.E_INVAL
    assert _call(g, w, None, 8, mu=0.9) == ap.E_INVAL
    assert _call(g, g + 4, v, 8) == ap.E_INVAL             # g and w partly overlap
    assert _call(g, w, w + 28, 8) == ap.E_INVAL            # w and v partly overlap
    assert _call(g, w, None, 0) == ap.OK                   # empty: nothing to do
    assert _call(None, None, None, 0) == ap.OK


# ------------------------------------------------------------------ GPU parity

torch = pytest.importorskip("torch")
DEV = torch.device("cuda:0")
gpu = pytest.mark.gpu
needs_gpu = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")


def inputs(d, seed):
    rng = np.random.default_rng(seed)
    g = (rng.standard_normal(d) * 1e-2).astype(np.float32)
    w = (rng.standard_normal(d) * 1e-1).astype(np.float32)
    v = (rng.standard_normal(d) * 1e-2).astype(np.float32)
    return g, w, v


def with_specials(g, w, v, seed):
    rng = np.random.default_rng(seed)
    d = g.size
    pick = lambda k: rng.choice(d, size=min(k, d), replace=False)
    g[pick(5)] = np.inf
    w[pick(5)] = -np.inf
    v[pick(5)] = np.nan
    g[pick(5)] = -0.0
    v[pick(5)] = np.float32(1e-41)                          # subnormal
    w[pick(5)] = np.float32(3e38)
    i = pick(20)
    g[i] = -np.float32(0.9) * v[i]                          # cancellation
    return g, w, v


def same(a, b):
    """bitwise equal, or NaN on both sides (NaN payloads may differ by platform)"""
    a, b = np.asarray(a, np.float32), np.asarray(b, np.float32)
    eq = a.view(np.uint32) == b.view(np.uint32)
    return bool(np.all(eq | (np.isnan(a) & np.isnan(b))))


def dev_slice(x, offset):
    """device copy of x starting `offset` floats into a fresh allocation"""
    base = torch.zeros(x.size + offset + 4, dtype=torch.float32, device=DEV)
    t = base[offset: offset + x.size]
    t.copy_(torch.from_numpy(x))
    return t


@gpu
@needs_gpu
@pytest.mark.parametrize("d", [1, 3, 4, 5, 1023, 4096, 4097, 65543, 1 << 20])
@pytest.mark.parametrize("mu", [0.9, 0.0])
@pytest.mark.parametrize("offset", [0, 1])
def test_sgd_parity(d, mu, offset):
    g, w, v = with_specials(*inputs(d, d + 17), seed=d)
    eta = 0.05
    gt, wt, vt = dev_slice(g, offset), dev_slice(w, offset), dev_slice(v, offset)
    ap.aspis_sgd(gt, wt, vt if mu else None, eta, mu)
    torch.cuda.synchronize()
    w_o, v_o = oracle.sgd(g, w, v if mu else None, eta, mu)
    assert same(wt.cpu().numpy(), w_o)
    if mu:
        assert same(vt.cpu().numpy(), v_o)
    else:
        assert same(vt.cpu().numpy(), v)                    # untouched


@gpu
@needs_gpu
def test_sgd_aliased_arrays():
    d = 10007
    g, w, v = inputs(d, 5)
    # g is also the momentum buffer: v <- mu*g + g, w <- w - eta*v
    gt, wt = dev_slice(g, 0), dev_slice(w, 0)
    ap.aspis_sgd(gt, wt, gt, 0.1, 0.9)
    torch.cuda.synchronize()
    v_o = oracle.sgd(g, np.zeros_like(g), g, 0.0, 0.9)[1]   # mu*g + g, alone
    w_o, _ = oracle.sgd(v_o, w, None, 0.1, 0.0)             # then w - eta*v
    assert same(gt.cpu().numpy(), v_o)
    assert same(wt.cpu().numpy(), w_o)


@gpu
@needs_gpu
def test_sgd_full_length_several_steps():
    d = synth.CONFIGS["k15_r3_d11m_strong_alie"].d           # ResNet-18 gradient length
    g, w, v = inputs(d, 3)
    gt, wt = dev_slice(g, 0), dev_slice(w, 0)
    vt = torch.zeros(d, dtype=torch.float32, device=DEV)
    v = np.zeros(d, np.float32)
    for step in range(3):
        eta = 0.1 * 0.95 ** step
        ap.aspis_sgd(gt, wt, vt, eta, 0.9)
        w, v = oracle.sgd(g, w, v, eta, 0.9)
    torch.cuda.synchronize()
    assert same(wt.cpu().numpy(), w)
    assert same(vt.cpu().numpy(), v)


@gpu
@needs_gpu
@pytest.mark.parametrize("name,d", [("k7_r3_d4096_alie", 4096), ("k15_r3_d1m_weak_reversed", 9001),
                                    ("k15_r3_d11m_strong_alie", 9001)])
def test_round_then_update(name, d):
    """Algorithm 1 end to end for three iterations: the round's median feeds
    the update; parameters and momentum match the oracle bit for bit."""
    wl = dataclasses.replace(synth.CONFIGS[name], d=d)
    oa = oracle.assign(wl.K, wl.r)
    host = synth.build_copies_np(wl, oa.file_workers)
    want = oracle.run_round(host, oa, wl.d, 0)
    a = ap.aspis_assign(wl.K, wl.r)
    copies = torch.from_numpy(host).to(DEV)
    buf = ap.RoundBuffers(a, wl.d, DEV)
    rng = np.random.default_rng(1)
    w = rng.standard_normal(wl.d).astype(np.float32)
    v = np.zeros(wl.d, np.float32)
    wt = torch.from_numpy(w).to(DEV)
    vt = torch.zeros(wl.d, dtype=torch.float32, device=DEV)
    for step in range(3):
        ap.aspis_round(copies, wl.d, a, buf.file_neq, buf.adj, buf.det, buf.sel, buf.out)
        ap.aspis_sgd(buf.out, wt, vt, 0.01, 0.9)
        w, v = oracle.sgd(want.out, w, v, 0.01, 0.9)
    torch.cuda.synchronize()
    assert same(buf.out.cpu().numpy(), want.out)
    assert same(wt.cpu().numpy(), w)
    assert same(vt.cpu().numpy(), v)
