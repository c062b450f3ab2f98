"""Proxy KV-cache decode step and append on the GPU against the float64 oracle.

Covers: both head widths, mixed cache fill (empty, partial, full capacity),
open blocks from empty to the last slot, batches beyond one 8-sequence GEMV
launch, single- and two-level append compression, the streaming rule (P
decode steps then an append), the paper-size decode (B = 8, d = 2048, 16 x 128
heads, 16384 cached proxies, 63 open tokens), and capacity errors that must
leave the offending sequence untouched, and the bulk prefill from a history
(gathered and in-place blocks, empty and sub-block histories, paper width).
"""
import numpy as np
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import decode as OD
from paper_2608_23463_gb300.decode import ProxyKVCache
from tests._util import assert_close, assert_grad_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


def _sync():
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)


def _np(t):
    return t.float().cpu().numpy()


def _check_step(spec, prm, st, cache):
    x = torch.from_numpy(st["x"]).to("cuda", torch.bfloat16)
    y = cache.step(x)
    _sync()
    ref_y, ref_st = OD.decode_step(spec, prm, st)
    assert_close("y", _np(y), ref_y)
    assert_grad_close("y - x", _np(y) - st["x"], ref_y - st["x"])
    for b in range(spec.batch):
        slot = int(st["n_open"][b])
        for k in ("X_open", "K_open", "V_open"):
            assert_close(f"{k}[{b}, {slot}]", _np(cache.s[k][b, slot]), ref_st[k][b, slot])
    assert (cache.s["n_open"].cpu().numpy() == ref_st["n_open"]).all()
    assert (cache.s["n_proxy"].cpu().numpy() == st["n_proxy"]).all()
    return ref_st


@pytest.mark.parametrize("d,dh,batch", [(256, 128, 3), (256, 64, 10), (192, 64, 2)])
def test_decode_step_matches_oracle(d, dh, batch):
    # d = 192: the split kernel's d/8 = 24 threads fill part of one warp
    spec = S.DecodeSpec(batch=batch, d=d, n_heads=d // dh, P=16, capacity=300)
    prm = S.make_decode_params(spec, 5)
    rng = np.random.default_rng(dh)
    n_proxy = rng.integers(0, 301, size=batch)
    n_proxy[0], n_proxy[-1] = 0, 300
    n_open = rng.integers(0, 16, size=batch)
    n_open[0], n_open[-1] = 0, 15
    st = S.make_decode_state(spec, 6, n_proxy, n_open)
    cache = ProxyKVCache(spec, prm, st)
    _check_step(spec, prm, st, cache)


def test_decode_step_paper_size():
    spec = S.spec_c4()
    prm = S.make_decode_params(spec, 3)
    st = S.make_decode_state(spec, 3, [spec.capacity] * 8, [63] * 8)
    cache = ProxyKVCache(spec, prm, st)
    _check_step(spec, prm, st, cache)


@pytest.mark.parametrize("levels", [1, 2])
def test_streaming_steps_then_append(levels):
    """P decode steps fill the open block; the append then writes the proxy
    the oracle computes from that block (Sec. 3.8), and the next step reads it."""
    P, d = 16, 256
    spec = S.DecodeSpec(batch=3, d=d, n_heads=2, P=P, levels=levels,
                        k1=4 if levels == 2 else 0, k2=4 if levels == 2 else 0, capacity=8)
    prm = S.make_decode_params(spec, 9)
    st = S.make_decode_state(spec, 10, [0, 3, 7], [0, 0, 0])
    cache = ProxyKVCache(spec, prm, st)
    rng = np.random.default_rng(11)
    for j in range(P):
        st = dict(st, x=S.round_bf16(rng.standard_normal((3, d)).astype(np.float32)))
        st = _check_step(spec, prm, st, cache)
        # carry the GPU's bf16 open rows forward, as the oracle's own state
        for k in ("X_open", "K_open", "V_open"):
            st[k] = _np(cache.s[k])
    H_in = rng.standard_normal((3, d)).astype(np.float32)
    cache.append(torch.from_numpy(H_in).cuda())
    _sync()
    ref = OD.kv_append(spec, prm, st, H_in)
    for b in range(3):
        row = int(st["n_proxy"][b])
        assert_close(f"K_proxy[{b}]", _np(cache.s["K_proxy"][b, row]), ref["K_proxy"][b, row])
        assert_close(f"V_proxy[{b}]", _np(cache.s["V_proxy"][b, row]), ref["V_proxy"][b, row])
    assert (cache.s["n_proxy"].cpu().numpy() == ref["n_proxy"]).all()
    assert (cache.s["n_open"].cpu().numpy() == 0).all()
    st = {k: (_np(v) if v.dtype == torch.bfloat16 else v.cpu().numpy()) for k, v in cache.s.items()}
    st["x"] = S.round_bf16(rng.standard_normal((3, d)).astype(np.float32))
    _check_step(spec, prm, st, cache)


def test_capacity_errors_leave_sequences_untouched():
    P, d = 16, 256
    spec = S.DecodeSpec(batch=3, d=d, n_heads=2, P=P, capacity=4)
    prm = S.make_decode_params(spec, 12)
    st = S.make_decode_state(spec, 13, [1, 2, 4], [3, P, 5])  # seq 1: open block full
    cache = ProxyKVCache(spec, prm, st)
    x = torch.from_numpy(st["x"]).to("cuda", torch.bfloat16)
    y = torch.full_like(x, 7.0)
    cache.step(x, y)
    with pytest.raises(pf.ProxyFormerError) as e:
        _sync()
    assert e.value.status == pf.PF_ERR_CAPACITY
    assert (y[1] == 7.0).all() and not (y[0] == 7.0).all()
    assert cache.s["n_open"].cpu().numpy().tolist() == [4, P, 6]
    # append: only sequence 1 has a full block, but sequence 2's cache is also full
    st2 = {k: (_np(v) if v.dtype == torch.bfloat16 else v.cpu().numpy()) for k, v in cache.s.items()}
    st2["n_open"] = np.array([P, P, P], np.int32)
    st2["n_proxy"] = np.array([0, 1, 4], np.int32)
    cache2 = ProxyKVCache(spec, prm, dict(st2, x=st["x"]))
    cache2.append()
    with pytest.raises(pf.ProxyFormerError) as e:
        _sync()
    assert e.value.status == pf.PF_ERR_CAPACITY
    assert cache2.s["n_proxy"].cpu().numpy().tolist() == [1, 2, 4]
    assert cache2.s["n_open"].cpu().numpy().tolist() == [0, 0, P]


def test_graph_replay_equals_direct_steps():
    """A captured step replays exactly like direct calls (the open-block
    counters advance on the device, so each replay fills the next slot)."""
    P, d = 16, 256
    spec = S.DecodeSpec(batch=3, d=d, n_heads=2, P=P, capacity=40)
    prm = S.make_decode_params(spec, 21)
    st = S.make_decode_state(spec, 22, [5, 0, 40], [0, 7, 14])
    direct, graphed = ProxyKVCache(spec, prm, st), ProxyKVCache(spec, prm, st)
    x = torch.from_numpy(st["x"]).to("cuda", torch.bfloat16)
    y1, y2 = torch.empty_like(x), torch.empty_like(x)
    g = graphed.capture_step(x, y2)
    for _ in range(2):
        direct.step(x, y1)
        g.replay()
        _sync()
        assert torch.equal(y1, y2)
    for k in direct.s:
        assert torch.equal(direct.s[k], graphed.s[k]), k
    assert graphed.s["n_open"].cpu().numpy().tolist() == [2, 9, 16]


_PREFILL_CASES = [
    # levels, batch, P blocks m, remainder r, capacity, with H_in
    (1, 3, 4, 5, 6, True),     # remainder with B > 1: blocks gathered first
    (2, 3, 4, 0, 4, False),    # m == capacity: one K/V GEMM over all sequences
    (2, 1, 3, 15, 10, True),   # one sequence: blocks read in place
    (1, 2, 0, 9, 3, False),    # shorter than a block: open block only
    (2, 2, 0, 0, 3, False),    # empty history
]


@pytest.mark.parametrize("levels,batch,m,r,cap,with_h", _PREFILL_CASES)
def test_prefill_matches_oracle(levels, batch, m, r, cap, with_h):
    """Bulk prefill (Sec. 3.8) against the oracle's: proxy K/V rows below m,
    open-block rows below r, counters m and r.  The cache starts full of
    unrelated rows, which prefill must overwrite from row 0."""
    P, d = 16, 256
    spec = S.DecodeSpec(batch=batch, d=d, n_heads=2, P=P, levels=levels,
                        k1=4 if levels == 2 else 0, k2=4 if levels == 2 else 0, capacity=cap)
    prm = S.make_decode_params(spec, 30 + levels)
    st0 = S.make_decode_state(spec, 31, [cap] * batch, [P - 1] * batch)
    cache = ProxyKVCache(spec, prm, st0)
    rng = np.random.default_rng(32)
    X = S.round_bf16(rng.standard_normal((batch, m * P + r, d)).astype(np.float32))
    H = rng.standard_normal((batch, m + (r > 0), d)).astype(np.float32) if with_h else None
    cache.prefill(torch.from_numpy(X).to("cuda", torch.bfloat16),
                  None if H is None else torch.from_numpy(H).cuda())
    _sync()
    ref = OD.kv_prefill(spec, prm, X, H)
    assert cache.s["n_proxy"].cpu().numpy().tolist() == [m] * batch
    assert cache.s["n_open"].cpu().numpy().tolist() == [r] * batch
    if m:
        for k in ("K_proxy", "V_proxy"):
            assert_close(k, _np(cache.s[k][:, :m]), ref[k][:, :m])
    if r:
        assert np.array_equal(_np(cache.s["X_open"][:, :r]), ref["X_open"][:, :r])
        for k in ("K_open", "V_open"):
            assert_close(k, _np(cache.s[k][:, :r]), ref[k][:, :r])
    # the next decode step reads the prefilled cache
    st = {k: (_np(v) if v.dtype == torch.bfloat16 else v.cpu().numpy()) for k, v in cache.s.items()}
    st["x"] = S.round_bf16(rng.standard_normal((batch, d)).astype(np.float32))
    _check_step(spec, prm, st, cache)


def test_prefill_paper_width():
    """d = 2048, 16 x 128 heads, P = 64 as 8 x 8 factors, eight sequences of
    3 blocks and 17 open tokens (a short history keeps the float64 oracle fast)."""
    spec = S.DecodeSpec(batch=8, d=2048, n_heads=16, P=64, levels=2, k1=8, k2=8, capacity=5)
    prm = S.make_decode_params(spec, 40)
    cache = ProxyKVCache(spec, prm, S.make_decode_state(spec, 41, [5] * 8, [0] * 8))
    rng = np.random.default_rng(42)
    X = S.round_bf16(rng.standard_normal((8, 3 * 64 + 17, 2048)).astype(np.float32))
    H = rng.standard_normal((8, 4, 2048)).astype(np.float32)  # 3 blocks + the partial one
    cache.prefill(torch.from_numpy(X).to("cuda", torch.bfloat16), torch.from_numpy(H).cuda())
    _sync()
    ref = OD.kv_prefill(spec, prm, X, H)
    for k in ("K_proxy", "V_proxy"):
        assert_close(k, _np(cache.s[k][:, :3]), ref[k][:, :3])
    assert np.array_equal(_np(cache.s["X_open"][:, :17]), ref["X_open"][:, :17])
    for k in ("K_open", "V_open"):
        assert_close(k, _np(cache.s[k][:, :17]), ref[k][:, :17])
    assert cache.s["n_proxy"].cpu().numpy().tolist() == [3] * 8
    assert cache.s["n_open"].cpu().numpy().tolist() == [17] * 8
