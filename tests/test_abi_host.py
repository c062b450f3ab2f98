"""Host-side checks of the C ABI (no GPU): the library builds, loads and exports
every entry point declared in include/proxyformer.h; descriptor validation and
workspace queries behave as documented."""
import ctypes
import os
import re

import pytest

import pf_synth as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pf():
    import paper_2608_23463_gb300 as pf
    from paper_2608_23463_gb300.buildlib import build
    build()
    pf.load()
    return pf


def declared_functions():
    txt = open(os.path.join(ROOT, "include", "proxyformer.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:pf_status|size_t|const char\s*\*|void|int|double)\s*\**\s*(\w+)\s*\(",
                                 txt, flags=re.M)))


def test_every_declared_symbol_is_exported(pf):
    names = declared_functions()
    assert len(names) >= 12, names
    lib = ctypes.CDLL(pf.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in proxyformer.h but not exported"
    assert set(names) == set(pf.EXPORTED)


def test_descriptor_validation(pf):
    ok = pf.layer_desc(S.spec_c3_layer(64))
    assert pf.proxy_layer_check(ok) == pf.PF_OK
    bad = pf.layer_desc(S.LayerSpec(batch=1, L=64, d=96, n_heads=1, P=4))
    assert pf.proxy_layer_check(bad) == pf.PF_ERR_INVALID_ARG
    bad = pf.layer_desc(S.LayerSpec(batch=1, L=64, d=128, n_heads=4, P=4))
    assert pf.proxy_layer_check(bad) == pf.PF_ERR_UNSUPPORTED  # head width 32
    bad = pf.layer_desc(S.LayerSpec(batch=1, L=64, d=128, n_heads=2, P=6, levels=2, k1=4, k2=2))
    assert pf.proxy_layer_check(bad) == pf.PF_ERR_INVALID_ARG
    assert "k1 * k2" in pf.pf_last_error()
    bad = pf.layer_desc(S.LayerSpec(batch=0, L=64, d=128, n_heads=2, P=4))
    assert pf.proxy_layer_check(bad) == pf.PF_ERR_INVALID_ARG


def test_variant_descriptor_validation(pf):
    """d_fine, the interaction F, RoPE and the cross injection are accepted
    exactly where they are built (1D bf16) and rejected elsewhere."""
    L = dict(batch=1, L=256, n_heads=2, P=16)
    check = lambda **kw: pf.proxy_layer_check(pf.layer_desc(S.LayerSpec(**{**L, **kw})))
    assert check(d=128, d_fine=64) == pf.PF_OK
    assert check(d=128, d_fine=32) == pf.PF_ERR_INVALID_ARG  # not a multiple of 64
    assert check(d=128, d_fine=64, dtype=S.F32) == pf.PF_ERR_UNSUPPORTED
    assert check(d=128, d_fine=64, inject=S.INJ_CROSS) == pf.PF_ERR_UNSUPPORTED
    assert check(d=128, inject=S.INJ_CROSS) == pf.PF_OK
    assert check(d=128, inject=S.INJ_CROSS, dtype=S.F32) == pf.PF_ERR_UNSUPPORTED
    assert check(d=128, interact=S.F_MLP) == pf.PF_OK
    assert check(d=128, interact=S.F_IDENTITY, mode=S.BIDIR_1D) == pf.PF_OK
    assert check(d=128, interact=3) == pf.PF_ERR_INVALID_ARG
    assert check(d=128, interact=S.F_MLP, dtype=S.F32) == pf.PF_ERR_UNSUPPORTED
    assert check(d=128, rope=1) == pf.PF_OK
    assert check(d=128, rope=1, interact=S.F_MLP) == pf.PF_ERR_INVALID_ARG
    s2d = S.spec_c5()
    assert pf.proxy_layer_check(pf.layer_desc(s2d)) == pf.PF_OK
    for kw in (dict(rope=1), dict(interact=S.F_IDENTITY), dict(d_fine=256)):
        bad = S.LayerSpec(**{**s2d.__dict__, **kw})
        assert pf.proxy_layer_check(pf.layer_desc(bad)) == pf.PF_ERR_UNSUPPORTED, kw
    # saved activations follow the variant: the MLP keeps its hidden layer,
    # identity drops Q/K/V, the cross injection keeps the token queries
    size = lambda **kw: pf.proxy_layer_saved_size(pf.layer_desc(S.LayerSpec(**{**L, **kw})))
    base = size(d=128)
    assert size(d=128, interact=S.F_IDENTITY) < base < size(d=128, interact=S.F_MLP)
    assert size(d=128, inject=S.INJ_CROSS) > 0
    assert size(d=128, d_fine=64) < base  # the decompressed update is d_fine wide


def test_sizes_scale_with_shape(pf):
    a = pf.layer_desc(S.LayerSpec(batch=1, L=4096, d=128, n_heads=2, P=16))
    b = pf.layer_desc(S.LayerSpec(batch=2, L=4096, d=128, n_heads=2, P=16))
    for f in (pf.proxy_layer_saved_size,
              lambda d: pf.proxy_layer_workspace_size(d, 1)):
        sa, sb = f(a), f(b)
        assert 0 < sa < sb
    # the saved buffer holds at least the decompressed update (bf16, L*d)
    assert pf.proxy_layer_saved_size(a) >= 4096 * 128 * 2
    # headline layer: saved ~ D (512 MiB) + Y + Z + proxy tensors
    big = pf.layer_desc(S.spec_c3_layer(64))
    assert 512 << 20 < pf.proxy_layer_saved_size(big) < 1 << 30


def test_calls_reject_bad_arguments_before_any_launch(pf):
    spec = S.LayerSpec(batch=1, L=256, d=128, n_heads=2, P=16)
    desc = pf.layer_desc(spec)
    prm = pf.layer_params({})
    with pytest.raises(pf.ProxyFormerError) as e:
        pf.proxy_layer_fwd(desc, prm, 16, None, None, 32, None, None, None, 0)
    assert e.value.status == pf.PF_ERR_INVALID_ARG
    full = pf.layer_params({k: 4096 for k in ("W_c1", "b_c1", "W_qkv", "W_o", "W_d1", "b_d1",
                                              "w_x", "w_dlt", "b_g")})
    with pytest.raises(pf.ProxyFormerError) as e:  # misaligned X
        pf.proxy_layer_fwd(desc, full, 8, None, None, 4096, None, None, 4096, 1 << 30)
    assert e.value.status == pf.PF_ERR_INVALID_ARG
    with pytest.raises(pf.ProxyFormerError) as e:  # workspace too small
        pf.proxy_layer_fwd(desc, full, 4096, None, None, 8192, None, None, 4096, 16)
    assert e.value.status == pf.PF_ERR_WORKSPACE
    with pytest.raises(pf.ProxyFormerError) as e:  # X_out aliases X
        pf.proxy_layer_fwd(desc, full, 4096, None, None, 4096, None, None, 4096, 1 << 30)
    assert e.value.status == pf.PF_ERR_INVALID_ARG
    with pytest.raises(pf.ProxyFormerError) as e:
        pf.pf_gemm_bf16(128, 100, 64, 4096, 0, 4096, 0, 4096, 100)
    assert e.value.status == pf.PF_ERR_INVALID_ARG


def test_prefill_rejects_bad_arguments_before_any_launch(pf):
    """proxy_layer_prefill / proxy_kv_prefill validate the cache descriptor
    against the layer, the capacity and the cache buffers on the host."""
    spec = S.LayerSpec(batch=2, L=100, d=128, n_heads=2, P=16)  # m = 6, r = 4
    desc = pf.layer_desc(spec)
    prm = pf.layer_params({})
    cache = pf.KVCache(*([4096] * 7))
    dp = pf.DecodeParams(*([4096] * 7))

    def call(cdesc, c=cache, d=dp, ldesc=desc):
        with pytest.raises(pf.ProxyFormerError) as e:
            pf.proxy_layer_prefill(ldesc, prm, cdesc, d, 4096, None, 8192, None, c, 4096, 1 << 30)
        return e.value.status

    ok = S.decode_spec_for_layer(spec, 6)
    mk = lambda ds: pf.DecodeDesc(ds.batch, ds.d, ds.n_heads, ds.P, ds.levels, ds.k1, ds.k2,
                                  ds.capacity)
    assert call(mk(S.decode_spec_for_layer(S.LayerSpec(batch=2, L=100, d=128, n_heads=2, P=8),
                                           6))) == pf.PF_ERR_INVALID_ARG  # other P
    assert call(mk(S.decode_spec_for_layer(spec, 5))) == pf.PF_ERR_CAPACITY
    assert call(mk(ok), c=pf.KVCache(*([4096] * 6 + [None]))) == pf.PF_ERR_INVALID_ARG
    assert call(mk(ok), d=pf.DecodeParams()) == pf.PF_ERR_INVALID_ARG  # r > 0 needs W_qkv
    s2d = S.spec_c5()
    assert call(mk(ok), ldesc=pf.layer_desc(s2d)) == pf.PF_ERR_UNSUPPORTED
    # the standalone prefill from a history
    ap = pf.AppendParams(*([4096] * 5))
    with pytest.raises(pf.ProxyFormerError) as e:
        pf.proxy_kv_prefill(mk(S.decode_spec_for_layer(spec, 5)), ap, dp, 4096, 100, None, cache,
                            4096, 1 << 30)
    assert e.value.status == pf.PF_ERR_CAPACITY
    with pytest.raises(pf.ProxyFormerError) as e:
        pf.proxy_kv_prefill(mk(ok), ap, dp, 4096, -1, None, cache, 4096, 1 << 30)
    assert e.value.status == pf.PF_ERR_INVALID_ARG
    assert pf.proxy_prefill_workspace_size(mk(ok), 100) > pf.proxy_prefill_workspace_size(mk(ok), 0)


def test_segments_plan_checks(pf):
    """Temporal-distance ratios: the segments must tile L, only the last may
    end mid-block, two levels need k1 * k2 == P per segment, and the layer
    must be batch 1, causal, bf16."""
    spec = S.LayerSpec(batch=1, L=300, d=128, n_heads=2, P=32)
    desc = pf.layer_desc(spec)
    ok = pf.segment_array([(256, 32), (44, 8)])
    assert pf.proxy_segments_saved_size(desc, ok) > 0
    assert pf.proxy_segments_workspace_size(desc, ok, 1) > 0
    assert pf.proxy_segments_saved_size(desc, pf.segment_array([(256, 32), (40, 8)])) == 0  # sum != L
    assert pf.proxy_segments_saved_size(desc, pf.segment_array([(250, 32), (50, 8)])) == 0  # mid-block
    two = pf.layer_desc(S.LayerSpec(batch=1, L=300, d=128, n_heads=2, P=32, levels=2, k1=8, k2=4))
    assert pf.proxy_segments_saved_size(two, pf.segment_array([(256, 32, 8, 4), (44, 8, 4, 2)])) > 0
    assert pf.proxy_segments_saved_size(two, pf.segment_array([(256, 32, 8, 8), (44, 8, 4, 2)])) == 0
    b2 = pf.layer_desc(S.LayerSpec(batch=2, L=300, d=128, n_heads=2, P=32))
    assert pf.proxy_segments_saved_size(b2, ok) == 0
    shared = pf.layer_params({})
    sp = pf.segment_params([{}, {}])
    with pytest.raises(pf.ProxyFormerError) as e:  # parameters missing: rejected on the host
        pf.proxy_segments_fwd(desc, ok, shared, sp, 4096, 8192, None, 4096, 1 << 30)
    assert e.value.status == pf.PF_ERR_INVALID_ARG
