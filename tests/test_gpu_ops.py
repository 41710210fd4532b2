"""Kernel-level parity through the C-ABI single-op entry points: the tcgen05 GEMM (all
epilogues, ragged M, both N tile widths), the CUDA-core GEMM, and flash attention
(self / shared-K/V cross, head_dim 64 and 128, ragged tails) against the oracle's fp64
primitives on the same bf16 inputs."""
import numpy as np
import pytest
import torch

from oracle import flashbon_oracle as O
from paper_2607_04461_gb300 import flashbon as fb
from paper_2607_04461_gb300 import synth
from _metrics import rel_max

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def model():
    fb.load_library()
    m = fb.Model(synth.TINY, synth.make_weights(synth.TINY))
    yield m
    m.close()


def randn(shape, seed, scale=1.0, dtype=torch.bfloat16):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(dtype).cuda()


def f64(t):
    return t.float().cpu().double().numpy()


GEMM_SHAPES = [
    (300, 256, 128),     # ragged M, BN=128, two K blocks
    (1, 128, 64),        # one row, one K block
    (2500, 384, 192),    # many tiles, BN=128
    (4000, 4608, 256),   # >= one tile per SM at BN=256 (the QKV shape's N)
    (640, 1536, 8960),   # long K (FFN down)
]


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_gemm_tc(model, M, N, K, epi):
    """Automatic choice: the 2-SM kernel when N % 256 == 0, else the 1-SM kernel."""
    _gemm_case(model, M, N, K, epi, impl=0)


@pytest.mark.parametrize("M,N,K", [(300, 256, 128), (1560, 1536, 1536), (513, 512, 8960)])
@pytest.mark.parametrize("epi", [0, 3])
def test_gemm_tc_1sm_forced(model, M, N, K, epi):
    _gemm_case(model, M, N, K, epi, impl=2)


@pytest.mark.parametrize("M", [1, 129, 256, 257, 1560, 49920])
def test_gemm_tc_2sm_ragged_rows(model, M):
    """Pair tiles of 256 rows: rows of the odd CTA may lie wholly past M."""
    _gemm_case(model, M, 512, 128, 0, impl=0)


# Stream-K shapes: the refine pass's one-candidate projections (1560 rows), a few tiles
# over a long K (13 pairs per tile), and two tiles over K = 9728 (about 38 pairs each).
SK_SHAPES = [(1560, 1536, 1536), (1560, 1536, 8960), (1560, 8960, 1536), (1560, 4608, 1536),
             (513, 512, 8960), (300, 256, 9728)]


@pytest.mark.parametrize("M,N,K", SK_SHAPES)
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_gemm_tc_stream_k_forced(model, M, N, K, epi):
    _gemm_case(model, M, N, K, epi, impl=4)


@pytest.mark.parametrize("M,N,K", SK_SHAPES[:2] + SK_SHAPES[-1:])
def test_gemm_stream_k_is_deterministic_and_matches_whole_tiles(model, M, N, K):
    """Cut tiles are summed in K order, so two runs agree bit for bit; whole-tile runs
    (impl 3) differ only by the fp32 summation order."""
    A = randn((M, K), 21)
    W = randn((N, K), 22, scale=K ** -0.5)
    resid = randn((M, N), 23, dtype=torch.float32)
    outs = []
    for impl in (4, 4, 3):
        out = torch.empty((M, N), dtype=torch.float32, device="cuda")
        fb.fb_op_gemm(model.handle, M, N, K, A, W, None, 2, out, resid, None, None, None, impl)
        outs.append(out)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1])
    assert rel_max(f64(outs[0]), f64(outs[2])) <= 1e-5


@pytest.mark.parametrize("M,N,K,twin", [
    (1560, 1536, 8960, 4),   # 42 tiles, 140 K blocks: stream-K
    (640, 1536, 8960, 4),    # 18 tiles, 140 K blocks: stream-K
    (1560, 1536, 1536, 3),   # 24 K blocks: whole tiles
    (49920, 1536, 8960, 3),  # more tiles than SM pairs: whole tiles
    (8192, 1536, 8960, 3),   # 2.5 rounds but A and W (166 MB) larger than half of L2
])
def test_gemm_automatic_stream_k_choice(model, M, N, K, twin):
    """impl 0 takes the stream-K split only for a long K under one wave of pair tiles: its
    result is bit-identical to the forced variant it chose."""
    A = randn((M, K), 51)
    W = randn((N, K), 52, scale=K ** -0.5)
    resid = randn((M, N), 53, dtype=torch.float32)
    outs = []
    for impl in (0, twin):
        out = torch.empty((M, N), dtype=torch.float32, device="cuda")
        fb.fb_op_gemm(model.handle, M, N, K, A, W, None, 2, out, resid, None, None, None, impl)
        outs.append(out)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1])


def test_gemm_stream_k_in_place_residual(model):
    M, N, K = 1560, 1536, 8960
    A, W = randn((M, K), 31), randn((N, K), 32, scale=K ** -0.5)
    h = randn((M, N), 33, dtype=torch.float32)
    h0 = f64(h)
    gate = randn((N,), 34, dtype=torch.float32)
    delta = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    fb.fb_op_gemm(model.handle, M, N, K, A, W, None, 3, h, h, gate, h, delta, 4)
    torch.cuda.synchronize()
    want = h0 + f64(gate) * O.linear(f64(A), f64(W))
    assert rel_max(f64(h), want) <= 1e-4
    assert rel_max(f64(delta), want - h0) <= 1e-2


@pytest.mark.parametrize("M,N,K", [(300, 256, 128), (300, 384, 9728)])
def test_gemm_stream_k_forced_rejects(model, M, N, K):
    """Too few K blocks per SM pair, or N not a multiple of 256: an error, no launch."""
    A, W = randn((M, K), 41), randn((N, K), 42)
    out = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(fb.FlashBonError) as e:
        fb.fb_op_gemm(model.handle, M, N, K, A, W, None, 0, out, None, None, None, None, 4)
    assert e.value.status == fb.FB_ECUDA
    _gemm_case(model, M, N, K, 0, impl=0)   # the model is still usable


@pytest.mark.parametrize("M,N,K", [(300, 256, 128), (77, 24, 40)])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_gemm_simt(model, M, N, K, epi):
    _gemm_case(model, M, N, K, epi, impl=1)


def _gemm_case(model, M, N, K, epi, impl):
    A = randn((M, K), 1)
    W = randn((N, K), 2, scale=K ** -0.5)
    bias = randn((N,), 3, dtype=torch.float32)
    resid = randn((M, N), 4, dtype=torch.float32)
    gate = randn((N,), 5, dtype=torch.float32)
    base = randn((M, N), 6, dtype=torch.float32)
    out = torch.empty((M, N), dtype=torch.bfloat16 if epi < 2 else torch.float32, device="cuda")
    delta = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, epi, out,
                  resid if epi >= 2 else None, gate if epi >= 2 else None,
                  base if epi == 3 else None, delta if epi == 3 else None, impl)
    torch.cuda.synchronize()
    y = O.linear(f64(A), f64(W), f64(bias))
    if epi == 0:
        assert rel_max(f64(out), y) <= 1e-2
    elif epi == 1:
        assert rel_max(f64(out), O.gelu_tanh(y)) <= 1e-2
    else:
        want = f64(resid) + f64(gate) * y
        assert rel_max(f64(out), want) <= 1e-4
        if epi == 3:
            assert rel_max(f64(delta), want - f64(base)) <= 1e-2


@pytest.mark.parametrize("M,N,K,impl", [
    (4999, 1536, 64, 0),     # the patch embedding: 2-SM kernel, one K block, ragged rows
    (3000, 128, 1536, 0),    # the padded head: 1-SM kernel, N = 128
    (300, 256, 128, 3),      # 2-SM whole tiles
    (1560, 1536, 8960, 4),   # 2-SM stream-K (cut tiles summed before the epilogue)
    (300, 256, 128, 2),      # 1-SM kernel forced
    (77, 24, 40, 1),         # CUDA-core kernel
])
@pytest.mark.parametrize("gated", [False, True])
def test_gemm_fp32_out_without_residual(model, M, N, K, impl, gated):
    """epi 2 with resid NULL: out = gate * (A W^T + bias) in fp32, every element written."""
    A = randn((M, K), 61)
    W = randn((N, K), 62, scale=K ** -0.5)
    bias = randn((N,), 63, dtype=torch.float32)
    gate = randn((N,), 64, dtype=torch.float32) if gated else None
    out = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, 2, out, None, gate, None, None, impl)
    torch.cuda.synchronize()
    y = O.linear(f64(A), f64(W), f64(bias))
    want = f64(gate) * y if gated else y
    assert not torch.isnan(out).any()
    assert rel_max(f64(out), want) <= 1e-4


def test_gemm_in_place_residual(model):
    """out == resid and base == out (the block's last GEMM runs this way)."""
    M, N, K = 257, 256, 128
    A, W = randn((M, K), 11), randn((N, K), 12, scale=K ** -0.5)
    h = randn((M, N), 13, dtype=torch.float32)
    h0 = f64(h)
    hb = randn((M, N), 14, dtype=torch.float32)
    delta = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    fb.fb_op_gemm(model.handle, M, N, K, A, W, None, 3, h, hb, None, h, delta)
    torch.cuda.synchronize()
    want = f64(hb) + O.linear(f64(A), f64(W))
    assert rel_max(f64(h), want) <= 1e-4
    assert rel_max(f64(delta), want - h0) <= 1e-2


ATTN_CASES = [
    # batch, Lq, Lkv, heads, dh, shared_kv
    (3, 150, 150, 2, 128, False),
    (2, 70, 40, 3, 64, True),
    (1, 1, 1, 1, 128, False),
    (2, 1560, 512, 2, 128, True),
    (1, 200, 333, 2, 64, False),
    (2, 1560, 1560, 2, 128, False),   # Wan2.1 self-attention length, ragged last tile
    (3, 256, 128, 1, 128, False),     # exact tile multiples
    (2, 129, 257, 2, 128, True),      # one row / one key past a tile
    # grids of more than one wave of 128-query CTAs take the persistent 256-query kernel
    # (P in TMEM)
    (4, 1560, 1560, 12, 128, False),
    (9, 600, 512, 12, 128, True),     # last CTA: tile A partly valid, tile B past Lq
    # the last key tile's MMAs cover only its 32-key chunks of real keys
    (2, 384, 192, 2, 128, False),     # 64 keys in the last tile; tile B starts at Lq
    (1, 300, 240, 2, 128, True),      # 112 keys: four chunks, the last one partial
    (2, 100, 193, 2, 128, False),     # 65 keys: three chunks
    # persistent 256-query CTAs: several items per CTA, one- and two-tile items mixed
    (12, 1560, 1560, 12, 128, False),
    (8, 300, 240, 12, 128, True),
]


@pytest.mark.parametrize("impl", [0, 3, 4], ids=["auto", "tc_q256", "tc_q256_persistent"])
def test_attention_large_logits(model, impl):
    """Scores spanning many powers of two exercise the rescaling of O."""
    batch, L, heads, dh = 2, 400, 2, 128
    D = heads * dh
    q = randn((batch * L, D), 41, scale=4.0)
    k = randn((batch * L, D), 42, scale=4.0)
    v = randn((batch * L, D), 43)
    o = torch.empty((batch * L, D), dtype=torch.bfloat16, device="cuda")
    fb.fb_op_attention(model.handle, q, D, k, D, v, D, o, D, batch, L, L, L, heads, dh, impl)
    torch.cuda.synchronize()
    qn, kn, vn, on = f64(q), f64(k), f64(v), f64(o)
    for b in range(batch):
        sl = slice(b * L, (b + 1) * L)
        want = O.attention(qn[sl].reshape(L, heads, dh), kn[sl].reshape(L, heads, dh),
                           vn[sl].reshape(L, heads, dh)).reshape(L, D)
        assert rel_max(on[sl], want) <= 2e-2


@pytest.mark.parametrize("impl", [0, 1, 2, 3, 4],
                         ids=["auto", "mma_sync", "tc_q128", "tc_q256", "tc_q256_persistent"])
@pytest.mark.parametrize("batch,Lq,Lkv,heads,dh,shared", ATTN_CASES)
def test_attention(model, batch, Lq, Lkv, heads, dh, shared, impl):
    D = heads * dh
    if impl >= 2 and dh != 128:
        z = torch.zeros((batch * max(Lq, Lkv), D), dtype=torch.bfloat16, device="cuda")
        with pytest.raises(fb.FlashBonError) as e:
            fb.fb_op_attention(model.handle, z, D, z, D, z, D, z, D, batch, Lq, Lkv, 0, heads,
                               dh, impl)
        assert e.value.status == fb.FB_EINVAL
        return
    q = randn((batch * Lq, D), 21)
    kvb = 1 if shared else batch
    k = randn((kvb * Lkv, D), 22)
    v = randn((kvb * Lkv, D), 23)
    o = torch.empty((batch * Lq, D), dtype=torch.bfloat16, device="cuda")
    fb.fb_op_attention(model.handle, q, D, k, D, v, D, o, D, batch, Lq, Lkv,
                       0 if shared else Lkv, heads, dh, impl)
    torch.cuda.synchronize()
    qn, kn, vn, on = f64(q), f64(k), f64(v), f64(o)
    for b in range(batch):
        kb = 0 if shared else b
        want = O.attention(qn[b * Lq:(b + 1) * Lq].reshape(Lq, heads, dh),
                           kn[kb * Lkv:(kb + 1) * Lkv].reshape(Lkv, heads, dh),
                           vn[kb * Lkv:(kb + 1) * Lkv].reshape(Lkv, heads, dh))
        got = on[b * Lq:(b + 1) * Lq]
        assert rel_max(got, want.reshape(Lq, D)) <= 2e-2
        assert np.abs(got - want.reshape(Lq, D)).mean() <= 2e-3


def test_attention_strided_qkv(model):
    """Self-attention reading q, k, v from one packed [rows][3D] buffer."""
    batch, L, heads, dh = 2, 97, 2, 128
    D = heads * dh
    qkv = randn((batch * L, 3 * D), 31)
    o = torch.empty((batch * L, D), dtype=torch.bfloat16, device="cuda")
    base = qkv.data_ptr()
    fb.fb_op_attention(model.handle, base, 3 * D, base + 2 * D, 3 * D, base + 4 * D, 3 * D, o,
                       D, batch, L, L, L, heads, dh)
    torch.cuda.synchronize()
    x = f64(qkv)
    for b in range(batch):
        r = x[b * L:(b + 1) * L]
        want = O.attention(r[:, :D].reshape(L, heads, dh), r[:, D:2 * D].reshape(L, heads, dh),
                           r[:, 2 * D:].reshape(L, heads, dh)).reshape(L, D)
        assert rel_max(f64(o)[b * L:(b + 1) * L], want) <= 2e-2


@pytest.mark.parametrize("ldo_pad,o_off", [(8, 0), (0, 8), (16, 0)],
                         ids=["row_stride_16B", "base_16B", "row_stride_32B"])
def test_attention_persistent_output_alignment(model, ldo_pad, o_off):
    """The persistent kernel stores O rows in 32-byte pieces only where the rows are
    32-byte aligned; a row stride or base aligned to 16 bytes only takes the 16-byte
    stores. Columns outside the heads' output stay untouched."""
    batch, L, heads, dh = 2, 300, 2, 128
    D = heads * dh
    ldo = D + ldo_pad
    q = randn((batch * L, D), 91)
    k = randn((batch * L, D), 92)
    v = randn((batch * L, D), 93)
    buf = torch.full((batch * L * ldo + o_off + 64,), 7.0, dtype=torch.bfloat16, device="cuda")
    o_ptr = buf.data_ptr() + 2 * o_off
    fb.fb_op_attention(model.handle, q, D, k, D, v, D, o_ptr, ldo, batch, L, L, L, heads, dh, 4)
    torch.cuda.synchronize()
    rows = buf[o_off:o_off + batch * L * ldo].view(batch * L, ldo)
    got = f64(rows[:, :D])
    if ldo_pad:
        assert torch.all(rows[:, D:] == 7.0)
    qn, kn, vn = f64(q), f64(k), f64(v)
    for b in range(batch):
        sl = slice(b * L, (b + 1) * L)
        want = O.attention(qn[sl].reshape(L, heads, dh), kn[sl].reshape(L, heads, dh),
                           vn[sl].reshape(L, heads, dh)).reshape(L, D)
        assert rel_max(got[sl], want) <= 2e-2


def test_pipe_probes_report_plausible_rates(model):
    """The measurement probes run and report values inside what the hardware allows: the
    tensor pipe at most 4096 MACs per SM clock (and at least half of it with no gap, less
    with a long gap), a special-function rate above zero and at most 64 per SM clock, and
    a TMEM load that takes clocks."""
    full = fb.fb_probe_mma_gap(0)
    gapped = fb.fb_probe_mma_gap(512)
    assert 2048 <= full <= 4096 * 1.01
    assert 0 < gapped < full
    for op in range(4):
        assert 0 < fb.fb_probe_mufu(op) <= 128
    for busy in (False, True):
        assert 10 < fb.fb_probe_tmem_load(busy) < 100000
    for form in range(14):
        for loaders, gap in ((0, 0), (7, 0)):
            assert 500 < fb.fb_probe_mma_mix(form, loaders, gap) < 4200
    with pytest.raises(fb.FlashBonError):
        fb.fb_probe_mma_mix(14)
    with pytest.raises(fb.FlashBonError):
        fb.fb_probe_mufu(4)
