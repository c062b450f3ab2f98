"""bench.py's accounting on the CPU: the algorithmic work that the roofline
fractions divide by, the compute peak at the sampled clock, and the DRAM
traffic lookup with its staleness rule.

The layer's FLOPs are re-derived here from the contractions of Alg. 1 one by
one (compression, the proxy interaction, decompression; every forward GEMM
has an input-gradient and a weight-gradient GEMM of its own size in the
backward; the attention backward re-forms S and dP and adds three more
products), not from the closed form bench.layer_work uses (Eq. complexity),
so a dropped or double-counted term in either shows up."""
import os

import pytest

import bench
import pf_synth as S


def _gemm_flops(shapes):
    return sum(2.0 * M * N * K for M, N, K in shapes)


def _layer_gemms(spec):
    """(M, N, K) of every forward contraction of one sequence (Alg. 1)."""
    L, d, P = spec.L, spec.d, spec.P
    m = -(-L // P)
    if spec.levels == 2:
        k1, k2 = spec.k1, spec.k2
        g = [(m * k2, d, k1 * d),          # level-1 compression: groups of k1 tokens
             (m, d, k2 * d)]               # level-2 compression: groups of k2 level-1 outputs
        g += [(m, 3 * d, d), (m, d, d)]    # Q, K, V and the output projection
        g += [(m, k2 * d, d),              # level-2 decompression
              (m * k2, k1 * d, d)]         # level-1 decompression, one row per k1 tokens
    else:
        g = [(m, d, P * d), (m, 3 * d, d), (m, d, d), (m, P * d, d)]
    return g


def _attention_pairs(m, causal):
    return sum(i + 1 for i in range(m)) if causal else m * m


@pytest.mark.parametrize("levels", [1, 2])
@pytest.mark.parametrize("mode", [0, 1])
def test_layer_flops_match_the_contractions(levels, mode):
    kw = dict(k1=8, k2=8) if levels == 2 else {}
    spec = S.LayerSpec(batch=2, L=262144 if levels == 2 else 65536, d=1024, n_heads=16, P=64,
                       levels=levels, mode=mode, **kw)
    m = -(-spec.L // spec.P)
    lin = _gemm_flops(_layer_gemms(spec))
    pairs = _attention_pairs(m, causal=(mode == 0))
    dh, nh = spec.d // spec.n_heads, spec.n_heads
    att_fwd = nh * pairs * (2 * dh + 2 * dh)                 # S = Q K^T, O = P V
    att_bwd = nh * pairs * (2 * dh * 5)                      # S again, dP, dV, dQ, dK
    fwd = spec.batch * (lin + att_fwd)
    bwd = spec.batch * (2 * lin + att_bwd)                   # dX and dW of every GEMM
    f_inf, _ = bench.layer_work(spec, train=False)
    f_train, _ = bench.layer_work(spec, train=True)
    assert f_inf == pytest.approx(fwd, rel=1e-12)
    assert f_train == pytest.approx(fwd + bwd, rel=1e-12)


def test_cross_and_mlp_layer_flops_match_the_contractions():
    """Gated cross injection (Eq. inj-cross with the gate of Sec. 3.7): the token-query
    and gate GEMM, the proxies' keys and values, the attention of every token
    over the proxies of earlier blocks, and the output projection replace the
    decompression; the single-proxy MLP replaces the attention by two GEMMs."""
    spec = S.LayerSpec(batch=1, L=262144, d=1024, n_heads=16, P=64, levels=2, k1=8, k2=8,
                       inject=S.INJ_CROSS)
    L, d, P, nh = spec.L, spec.d, spec.P, spec.n_heads
    m = L // P
    g = _layer_gemms(spec)[:4]                               # compressions, QKV, O
    g += [(L, d + nh, d), (m, 2 * d, d), (L, d, d)]         # [Q | gate], [K | V], output
    vis = sum(P * b for b in range(m))                       # token in block b sees b proxies
    att = 4.0 * d * (_attention_pairs(m, True) + vis)
    lin = _gemm_flops(g)
    assert bench.layer_work(spec)[0] == pytest.approx(3 * lin + 3.5 * att, rel=1e-12)

    mlp = S.LayerSpec(batch=1, L=262144, d=1024, n_heads=16, P=64, levels=2, k1=8, k2=8,
                      interact=S.F_MLP)
    g = [x for x in _layer_gemms(mlp) if x not in ((m, 3 * d, d), (m, d, d))]
    g += [(m, 4 * d, d), (m, d, 4 * d)]
    assert bench.layer_work(mlp)[0] == pytest.approx(3 * _gemm_flops(g), rel=1e-12)


def test_2d_layer_flops_match_the_contractions():
    """2D layer (Sec. 3.9): each 8 x 8 patch of tokens compressed to a proxy,
    bidirectional attention over the patch grid, and the decompression to a
    scale and a shift per token channel (affine injection, 2 P d_fine wide)."""
    spec = S.spec_c5()
    d, P = spec.d, spec.P
    m = spec.L // P
    g = [(m, d, P * d), (m, 3 * d, d), (m, d, d), (m, 2 * P * d, d)]
    att = 4.0 * d * m * m
    expect = spec.batch * (3 * _gemm_flops(g) + 3.5 * att)
    assert bench.layer_work(spec)[0] == pytest.approx(expect, rel=1e-12)


def test_headline_work_and_roofline_time():
    """The benchmark layer (L = 262144, d = 1024, P = 64 as 8 x 8): 3.934
    TFLOP and 3.52 GB per fwd+bwd step; X, dX_out read and X_out, dX written
    once, X read once more by the injection and once by the backward, the
    weights read once per pass and their fp32 gradients written once."""
    spec = S.spec_c3_layer(64)
    flops, nbytes = bench.layer_work(spec)
    assert flops == pytest.approx(3.934e12, rel=1e-3)
    act = spec.batch * spec.L * spec.d * 2
    d, k1, k2 = spec.d, spec.k1, spec.k2
    weights = k1 * d * d + k2 * d * d + 4 * d * d + k2 * d * d + k1 * d * d
    assert nbytes == pytest.approx(6 * act + 2 * 2 * weights + 4 * weights, rel=1e-12)
    assert nbytes == pytest.approx(3.52e9, rel=2e-3)
    # at the measured burst peak the step cannot take less than ~2.04 ms
    assert flops / 1926.3e12 * 1e3 == pytest.approx(2.042, abs=2e-3)


def test_compute_peak_follows_the_sampled_clock():
    peaks = {"bf16_tflops": 1926.3}
    assert bench.compute_peak(peaks, None)[0] == 1926.3
    assert bench.compute_peak(peaks, {"sm_mhz": 2070, "sm_max_mhz": 2070})[0] == 1926.3
    p, src = bench.compute_peak(peaks, {"sm_mhz": 1035, "sm_max_mhz": 2070})
    assert p == pytest.approx(1926.3 / 2) and "1035/2070" in src
    # a sample above the maximum never raises the peak above the burst figure
    assert bench.compute_peak(peaks, {"sm_mhz": 2100, "sm_max_mhz": 2070})[0] == 1926.3


def test_config_entry_takes_the_larger_bound():
    peaks = {"bf16_tflops": 1000.0, "hbm_gbs": 5000.0}
    dom = {"kernel": "k"}
    # 1 TFLOP at 1000 TFLOP/s = 1 ms against 1 GB at 5000 GB/s = 0.2 ms: tensor-bound
    e = bench.config_entry("m", 1000, 2.0, (1e12, 1e9), dom, peaks, 5)
    assert e["roofline"]["bound"] == "tensor"
    assert e["roofline"]["frac"] == pytest.approx(0.5)
    assert e["value"] == pytest.approx(1000 / 2e-3)
    # 10 GB at 5000 GB/s = 2 ms against 1 ms of FLOPs: HBM-bound
    e = bench.config_entry("m", 1000, 4.0, (1e12, 1e10), dom, peaks, 5)
    assert e["roofline"]["bound"] == "hbm" and e["roofline"]["frac"] == pytest.approx(0.5)
    # an fp32 workload divides by the measured FFMA peak and says "alu"
    e = bench.config_entry("m", 1000, 2.0, (50e9, 1e6), dom, peaks, 5, ffma=50.0)
    assert e["roofline"]["bound"] == "alu" and e["roofline"]["frac"] == pytest.approx(0.5)


def test_traffic_lookup_scales_by_tokens_and_drops_stale_captures(tmp_path, monkeypatch):
    label = "decompress_d1_inject"
    (tmp_path / "profiles").mkdir()
    csrc = os.path.join(bench.ROOT, "paper_2608_23463_gb300", "csrc")
    (tmp_path / "paper_2608_23463_gb300").mkdir()
    os.symlink(csrc, tmp_path / "paper_2608_23463_gb300" / "csrc")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h = bench.source_hash(label)
    (tmp_path / "profiles" / "traffic.txt").write_text(
        "# label bytes units hash\n%s 1000 100 %s\ninj_bwd 5 1 0000000000000000\n" % (label, h))
    assert bench.traffic_from_profile(label, 400) == pytest.approx(4000.0)
    assert bench.traffic_from_profile("inj_bwd", 1) is None       # captured at other sources
    assert bench.traffic_from_profile("attn_fwd", 1) is None      # never captured
    # every label hashes the files that define its kernel
    assert "gemm_tc.cuh" in bench.kernel_files(label)
    assert "elementwise.cu" in bench.kernel_files("inj_bwd")
    assert "attention_tc.cu" in bench.kernel_files("attn_fwd")


@pytest.mark.parametrize("levels", [1, 2])
def test_one_segment_has_the_work_of_the_layer(levels):
    """Temporal-distance ratios (Sec. 3.6) with a single segment are the
    ordinary layer, work included; with several, each segment's compression
    and decompression at its own ratio plus one attention over all proxies."""
    kw = dict(k1=8, k2=8) if levels == 2 else {}
    seg = [(262144, 64, 8, 8)]
    lay = S.LayerSpec(batch=1, L=262144, d=1024, n_heads=16, P=64, levels=levels, **kw)
    f, b = bench.segments_work(1024, 16, levels, seg)
    fl, bl = bench.layer_work(lay)
    assert f == pytest.approx(fl, rel=1e-12) and b == pytest.approx(bl, rel=1e-12)
    segs = [(131072, 256, 16, 16), (98304, 64, 8, 8), (32768, 16, 4, 4)]
    f3, _ = bench.segments_work(1024, 16, 2, segs)
    m_tot = sum(Ls // Ps for Ls, Ps, _, _ in segs)
    lin = 0.0
    for Ls, Ps, a, c in segs:
        sp = S.LayerSpec(batch=1, L=Ls, d=1024, n_heads=16, P=Ps, levels=2, k1=a, k2=c)
        lin += _gemm_flops([x for x in _layer_gemms(sp)
                            if x not in ((Ls // Ps, 3 * 1024, 1024), (Ls // Ps, 1024, 1024))])
    lin += _gemm_flops([(m_tot, 3 * 1024, 1024), (m_tot, 1024, 1024)])
    att = 4.0 * 1024 * _attention_pairs(m_tot, True)
    assert f3 == pytest.approx(3 * lin + 3.5 * att, rel=1e-12)


def test_decode_step_bytes():
    """Decode at the paper's shape (B = 8, d = 2048, 16384 cached proxies):
    ~1.11 GB per step, almost all of it the cached K and V rows, which every
    step streams once; the weights add 4.125 d^2 bf16 elements."""
    spec = S.spec_c4()
    b = bench.decode_step_bytes(spec, 128)
    cache = spec.batch * spec.capacity * 2 * spec.d * 2
    assert b == pytest.approx(1.1105e9, rel=1e-3)
    assert cache / b > 0.96
    assert b - bench.decode_step_bytes(spec, 1) == pytest.approx(
        spec.batch * (32.5 - 1.0) * 2 * spec.d * 2)  # the open block's mean fill
