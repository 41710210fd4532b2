"""The allocation-free stream-K GEMM entry point against the model's stream-K GEMM
(fb_op_gemm, impl 4): the same partition of the same units in the same K order, so the
results agree bit for bit, on two calls in a row (the static counters must be back at
zero after each call). Collected last, so it also runs after every other GPU test."""
import pytest
import torch

from paper_2607_04461_gb300 import flashbon as fb
from paper_2607_04461_gb300 import synth

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


@pytest.mark.parametrize("M,N,K,epi", [(1560, 1536, 1536, 2), (1560, 1536, 8960, 3),
                                       (1560, 8960, 1536, 1), (300, 256, 9728, 0)])
def test_noalloc_matches_op_gemm_on_two_calls_in_a_row(model, M, N, K, epi):
    A, W = randn((M, K), 1), randn((N, K), 2, scale=K ** -0.5)
    bias, gate = randn((N,), 3, dtype=torch.float32), randn((N,), 4, dtype=torch.float32)
    resid = randn((M, N), 5, dtype=torch.float32) if epi >= 2 else None
    base = randn((M, N), 6, dtype=torch.float32) if epi == 3 else None
    odt = torch.bfloat16 if epi < 2 else torch.float32

    def outs():
        o = torch.empty((M, N), dtype=odt, device="cuda")
        d = torch.empty((M, N), dtype=torch.bfloat16, device="cuda") if epi == 3 else None
        return o, d
    ref, ref_d = outs()
    fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, epi, ref, resid,
                  gate if epi >= 2 else None, base, ref_d, 4)
    stream = torch.cuda.current_stream().cuda_stream
    got = []
    for _ in range(2):
        o, d = outs()
        torch.cuda.synchronize()
        fb.fb_gemm_streamk_noalloc(stream, M, N, K, A, W, bias, epi, o, resid,
                                   gate if epi >= 2 else None, base, d)
        got.append((o, d))
    torch.cuda.synchronize()
    for o, d in got:
        assert torch.equal(o, ref)
        if epi == 3:
            assert torch.equal(d, ref_d)


def test_noalloc_allocates_nothing_per_call():
    M, N, K = 1560, 1536, 1536
    A, W = randn((M, K), 11), randn((N, K), 12, scale=K ** -0.5)
    out = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    call = lambda: fb.fb_gemm_streamk_noalloc(None, M, N, K, A, W, None, 0, out)  # noqa: E731
    call()   # the first call on a device may load the library's static device arrays
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        call()
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


@pytest.mark.parametrize("M,N,K", [(300, 256, 128), (300, 384, 9728), (300, 256, 100)])
def test_noalloc_rejects_what_it_cannot_run(M, N, K):
    A, W = randn((M, K), 21), randn((N, K), 22)
    out = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(fb.FlashBonError) as e:
        fb.fb_gemm_streamk_noalloc(None, M, N, K, A, W, None, 0, out)
    assert e.value.status == fb.FB_EINVAL
    with pytest.raises(fb.FlashBonError) as e:
        fb.fb_gemm_streamk_noalloc(None, M, N, K, None, W, None, 0, out)
    assert e.value.status == fb.FB_EINVAL


def test_noalloc_wait_timeout_clears_its_counters(model):
    """With the static tile counters poisoned (a large negative count, as a crashed launch
    could leave them) a finisher waits for a count no launch reaches. With a short device
    wait limit the call returns FB_ECUDA "device wait timed out"; it must leave the
    counters at zero, so the next two calls match fb_op_gemm impl 4 bit for bit."""
    M, N, K, epi = 1560, 1536, 8960, 2
    A, W = randn((M, K), 31), randn((N, K), 32, scale=K ** -0.5)
    bias, gate = randn((N,), 33, dtype=torch.float32), randn((N,), 34, dtype=torch.float32)
    resid = randn((M, N), 35, dtype=torch.float32)
    ref = torch.empty((M, N), dtype=torch.float32, device="cuda")
    fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, epi, ref, resid, gate, None, None, 4)
    out = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    fb.fb_test_poison_counters(None)
    fb.fb_set_device_wait_limit(20_000_000)
    try:
        with pytest.raises(fb.FlashBonError) as e:
            fb.fb_gemm_streamk_noalloc(None, M, N, K, A, W, bias, epi, out, resid, gate)
    finally:
        fb.fb_set_device_wait_limit(0)
    assert e.value.status == fb.FB_ECUDA and "device wait timed out" in str(e.value)
    for _ in range(2):
        o = torch.empty((M, N), dtype=torch.float32, device="cuda")
        fb.fb_gemm_streamk_noalloc(None, M, N, K, A, W, bias, epi, o, resid, gate)
        torch.cuda.synchronize()
        assert torch.equal(o, ref)
