"""ctypes binding of libflashbon.so (include/flashbon.h). Argument marshalling only:
every step of the draft path runs in the library's CUDA kernels. There is no CPU
fallback: if the library is missing, loading raises.

Buffers may be numpy arrays (host memory) or torch tensors (host or CUDA); they are
passed to the library as raw pointers and must be contiguous float32 / uint8 / int32.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import synth

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libflashbon.so")

FB_OK, FB_EINVAL, FB_ENOMEM, FB_ECUDA, FB_EPLAN, FB_ESTATE = range(6)
KERNEL_KINDS = ["gemm_tc", "gemm_simt", "attn_self", "attn_cross", "ln_mod", "qk_norm_rope",
                "proxy_add", "patch_embed", "head_euler", "small"]
K = {name: i for i, name in enumerate(KERNEL_KINDS)}


class FlashBonError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"flashbon status {status}: {msg}")
        self.status = status


class fb_cfg(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in (
        "depth", "dim", "heads", "head_dim", "ffn", "text_len", "text_dim", "latent_c",
        "latent_h", "latent_w", "patch", "max_n", "freq_dim")] + [
        ("eps_ln", ctypes.c_float), ("eps_rms", ctypes.c_float), ("rope_theta", ctypes.c_float)]


class fb_sampler_opts(ctypes.Structure):
    _fields_ = [("guidance", ctypes.c_float), ("text_uncond", ctypes.c_void_p),
                ("sde_a", ctypes.c_float), ("noise", ctypes.c_void_p),
                ("keep_state", ctypes.c_int), ("state", ctypes.c_void_p),
                ("warm_steps", ctypes.c_int)]


class fb_kstat(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_uint64), ("ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


EXPORTS = ["fb_weights_count", "fb_weights_entry", "fb_init_model", "fb_free", "fb_set_stream",
           "fb_encode_text", "fb_draft", "fb_refine", "fb_plan_from_phi", "fb_block_forward",
           "fb_last_error", "fb_set_timing", "fb_get_stats", "fb_reset_stats", "fb_kernel_name",
           "fb_op_gemm", "fb_op_attention", "fb_draft_ex", "fb_refine_ex", "fb_select_elo",
           "fb_set_op_repeat", "fb_gemm_streamk_noalloc", "fb_state_bytes", "fb_state_offload",
           "fb_state_wait", "fb_set_sm_budget", "fb_sm_split_create", "fb_sm_split_info",
           "fb_sm_split_free", "fb_pipeline_step", "fb_set_device_wait_limit",
           "fb_test_fail_alloc", "fb_test_alloc_calls", "fb_test_poison_counters",
           "fb_probe_mma_rate", "fb_probe_mma_gap", "fb_probe_mufu", "fb_probe_tmem_load",
           "fb_probe_mma_mix"]

PAIR_VERIFIER = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                 ctypes.POINTER(ctypes.c_int))

_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Loads libflashbon.so (raises FileNotFoundError if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise FileNotFoundError(f"{path} not built: run paper_2607_04461_gb300.build.build()")
    L = ctypes.CDLL(path)
    P, I, S, F, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float, ctypes.c_double
    sig = {
        "fb_weights_count": (I, [ctypes.POINTER(fb_cfg), ctypes.POINTER(I), ctypes.POINTER(S)]),
        "fb_weights_entry": (I, [ctypes.POINTER(fb_cfg), I, ctypes.POINTER(ctypes.c_char_p),
                                 ctypes.POINTER(S), ctypes.POINTER(S)]),
        "fb_init_model": (I, [ctypes.POINTER(fb_cfg), P, ctypes.POINTER(P)]),
        "fb_free": (None, [P]),
        "fb_set_stream": (I, [P, P]),
        "fb_encode_text": (I, [P, P]),
        "fb_draft": (I, [P, P, I, P, P, I, P, P]),
        "fb_refine": (I, [P, P, P, P, I]),
        "fb_draft_ex": (I, [P, P, I, P, P, I, P, P, ctypes.POINTER(fb_sampler_opts)]),
        "fb_refine_ex": (I, [P, P, P, P, I, ctypes.POINTER(fb_sampler_opts)]),
        "fb_select_elo": (I, [P, I, D, D, D, D, PAIR_VERIFIER, P, ctypes.POINTER(I),
                              ctypes.POINTER(ctypes.c_double), ctypes.POINTER(I)]),
        "fb_plan_from_phi": (I, [I, I, I, I, I, I, I, I, P, P]),
        "fb_block_forward": (I, [P, I, P, I, F]),
        "fb_last_error": (ctypes.c_char_p, []),
        "fb_set_timing": (I, [P, I]),
        "fb_set_op_repeat": (I, [P, I]),
        "fb_get_stats": (I, [P, P]),
        "fb_reset_stats": (I, [P]),
        "fb_kernel_name": (ctypes.c_char_p, [I]),
        "fb_op_gemm": (I, [P, I, I, I, P, P, P, I, P, P, P, P, P, I]),
        "fb_op_attention": (I, [P, P, I, P, I, P, I, P, I, I, I, I, I, I, I, I]),
        "fb_gemm_streamk_noalloc": (I, [P, I, I, I, P, P, P, I, P, P, P, P, P]),
        "fb_state_bytes": (I, [P, ctypes.POINTER(S)]),
        "fb_state_offload": (I, [P, I, I, ctypes.POINTER(P)]),
        "fb_state_wait": (I, [P]),
        "fb_set_sm_budget": (I, [P, I]),
        "fb_sm_split_create": (I, [I, ctypes.POINTER(P)]),
        "fb_sm_split_info": (I, [P, I, ctypes.POINTER(P), ctypes.POINTER(I)]),
        "fb_sm_split_free": (None, [P]),
        "fb_pipeline_step": (I, [P, P, I, P, P, I, P, P, ctypes.POINTER(fb_sampler_opts),
                                 P, P, P, I, ctypes.POINTER(fb_sampler_opts)]),
        "fb_set_device_wait_limit": (I, [ctypes.c_ulonglong]),
        "fb_test_fail_alloc": (I, [ctypes.c_long]),
        "fb_test_alloc_calls": (ctypes.c_long, []),
        "fb_test_poison_counters": (I, [P]),
        "fb_probe_mma_rate": (I, [I, I, I, ctypes.POINTER(ctypes.c_double)]),
        "fb_probe_mma_gap": (I, [I, ctypes.POINTER(ctypes.c_double)]),
        "fb_probe_mufu": (I, [I, ctypes.POINTER(ctypes.c_double)]),
        "fb_probe_tmem_load": (I, [I, ctypes.POINTER(ctypes.c_double)]),
        "fb_probe_mma_mix": (I, [I, I, I, ctypes.POINTER(ctypes.c_double)]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype, fn.argtypes = res, args
    _lib = L
    return L


def _check(status):
    if status != FB_OK:
        raise FlashBonError(status, load_library().fb_last_error().decode())


def _ptr(x, dtype=None):
    """Raw pointer of a numpy array or torch tensor (must be contiguous)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if dtype is not None and x.dtype != dtype:
            raise TypeError(f"expected {dtype}, got {x.dtype}")
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("array must be C-contiguous")
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return x.data_ptr()
    if isinstance(x, int):
        return x
    raise TypeError(f"unsupported buffer type {type(x)}")


def make_cfg(cfg: synth.Cfg) -> fb_cfg:
    c = fb_cfg()
    for f, _ in fb_cfg._fields_:
        setattr(c, f, getattr(cfg, f))
    return c


def pack_weights(cfg: synth.Cfg, weights: dict):
    """Packs named weights into the library's fp32 layout (fb_weights_entry order): a
    numpy buffer, or a CUDA tensor when the weights are CUDA tensors."""
    L = load_library()
    c = make_cfg(cfg)
    count, total = ctypes.c_int(), ctypes.c_size_t()
    _check(L.fb_weights_count(ctypes.byref(c), ctypes.byref(count), ctypes.byref(total)))
    first = next(iter(weights.values()))
    if getattr(first, "is_cuda", False):
        import torch
        buf = torch.empty(total.value, dtype=torch.float32, device=first.device)
        name, off, numel = ctypes.c_char_p(), ctypes.c_size_t(), ctypes.c_size_t()
        for i in range(count.value):
            _check(L.fb_weights_entry(ctypes.byref(c), i, ctypes.byref(name),
                                      ctypes.byref(off), ctypes.byref(numel)))
            w = weights[name.value.decode()].reshape(-1)
            if w.numel() != numel.value:
                raise ValueError(f"{name.value.decode()}: {w.numel()} elements, "
                                 f"expected {numel.value}")
            buf[off.value: off.value + numel.value].copy_(w)
        return buf
    buf = np.empty(total.value, np.float32)
    name, off, numel = ctypes.c_char_p(), ctypes.c_size_t(), ctypes.c_size_t()
    for i in range(count.value):
        _check(L.fb_weights_entry(ctypes.byref(c), i, ctypes.byref(name), ctypes.byref(off),
                                  ctypes.byref(numel)))
        w = np.asarray(weights[name.value.decode()], np.float32).ravel()
        if w.size != numel.value:
            raise ValueError(f"{name.value.decode()}: {w.size} elements, expected {numel.value}")
        buf[off.value: off.value + numel.value] = w
    return buf


# ---- functions with the C-ABI names -------------------------------------------------

def fb_init_model(cfg: synth.Cfg, weights) -> int:
    """weights: dict of named arrays, or an already packed fp32 buffer."""
    L = load_library()
    packed = weights if isinstance(weights, np.ndarray) or hasattr(weights, "data_ptr") \
        else pack_weights(cfg, weights)
    c = make_cfg(cfg)
    h = ctypes.c_void_p()
    _check(L.fb_init_model(ctypes.byref(c), _ptr(packed, np.float32), ctypes.byref(h)))
    return h.value


def fb_free(model: int) -> None:
    load_library().fb_free(model)


def fb_set_stream(model: int, stream) -> None:
    """stream: a torch.cuda.Stream, a raw cudaStream_t int, or None (model's own)."""
    s = getattr(stream, "cuda_stream", stream)
    _check(load_library().fb_set_stream(model, s))


def fb_set_sm_budget(model: int, n_sms: int) -> None:
    _check(load_library().fb_set_sm_budget(model, int(n_sms)))


class SmSplit:
    """Two disjoint SM partitions of the current device (green contexts), each with its
    own stream: part 0 holds n_sms SMs, part 1 the rest. streams[i] is a raw
    cudaStream_t handle (int) for Model.set_stream; sms[i] the part's SM count."""

    def __init__(self, n_sms: int):
        L = load_library()
        h = ctypes.c_void_p()
        _check(L.fb_sm_split_create(int(n_sms), ctypes.byref(h)))
        self.handle = h.value
        self.streams, self.sms = [], []
        for part in (0, 1):
            st, n = ctypes.c_void_p(), ctypes.c_int()
            _check(L.fb_sm_split_info(self.handle, part, ctypes.byref(st), ctypes.byref(n)))
            self.streams.append(st.value)
            self.sms.append(n.value)

    def close(self):
        if self.handle:
            load_library().fb_sm_split_free(self.handle)
            self.handle = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def fb_encode_text(model: int, text_ctx) -> None:
    _check(load_library().fb_encode_text(model, _ptr(text_ctx, np.float32)))


def fb_draft(model: int, latents, n: int, text_ctx, schedule, skip_mask=None,
             proxy_plan=None) -> None:
    sched = np.ascontiguousarray(schedule, np.float32)
    sk = None if skip_mask is None else np.ascontiguousarray(skip_mask, np.uint8)
    px = None if proxy_plan is None else np.ascontiguousarray(proxy_plan, np.int32)
    n_steps = len(sched) - 1
    for a in (sk, px):
        if a is not None and a.shape[0] != n_steps:
            raise ValueError("plan rows must equal len(schedule) - 1")
    _check(load_library().fb_draft(model, _ptr(latents, np.float32), n,
                                   _ptr(text_ctx, np.float32), _ptr(sched), n_steps,
                                   _ptr(sk), _ptr(px)))


def fb_refine(model: int, latent, text_ctx, full_schedule) -> None:
    sched = np.ascontiguousarray(full_schedule, np.float32)
    _check(load_library().fb_refine(model, _ptr(latent, np.float32), _ptr(text_ctx, np.float32),
                                    _ptr(sched), len(sched) - 1))


def make_opts(guidance=1.0, text_uncond=None, sde_a=0.0, noise=None, keep_state=False,
              state=None, warm_steps=0):
    """fb_sampler_opts; keeps references to the buffers it points to. state is a cached
    state buffer (fb_state_offload layout: numpy uint8 array or torch tensor)."""
    o = fb_sampler_opts(float(guidance), _ptr(text_uncond, np.float32), float(sde_a),
                        _ptr(noise, np.float32), int(bool(keep_state)), _ptr(state),
                        int(warm_steps))
    o._keep = (text_uncond, noise, state)
    return o


def fb_state_bytes(model) -> int:
    n = ctypes.c_size_t()
    _check(load_library().fb_state_bytes(model, ctypes.byref(n)))
    return n.value


def fb_state_offload(model, first: int, dsts) -> None:
    """Starts the copies of candidates first .. first + len(dsts) - 1's cached states into
    dsts (fb_state_bytes bytes each; pinned host memory lets them overlap later work);
    fb_state_wait waits for them."""
    arr = (ctypes.c_void_p * len(dsts))(*[_ptr(d) for d in dsts])
    _check(load_library().fb_state_offload(model, first, len(dsts), arr))


def fb_state_wait(model) -> None:
    _check(load_library().fb_state_wait(model))


def fb_draft_ex(model: int, latents, n: int, text_ctx, schedule, skip_mask=None,
                proxy_plan=None, opts=None) -> None:
    sched = np.ascontiguousarray(schedule, np.float32)
    sk = None if skip_mask is None else np.ascontiguousarray(skip_mask, np.uint8)
    px = None if proxy_plan is None else np.ascontiguousarray(proxy_plan, np.int32)
    _check(load_library().fb_draft_ex(model, _ptr(latents, np.float32), n,
                                      _ptr(text_ctx, np.float32), _ptr(sched), len(sched) - 1,
                                      _ptr(sk), _ptr(px),
                                      None if opts is None else ctypes.byref(opts)))


def fb_refine_ex(model: int, latent, text_ctx, full_schedule, opts=None) -> None:
    sched = np.ascontiguousarray(full_schedule, np.float32)
    _check(load_library().fb_refine_ex(model, _ptr(latent, np.float32),
                                       _ptr(text_ctx, np.float32), _ptr(sched), len(sched) - 1,
                                       None if opts is None else ctypes.byref(opts)))


def fb_pipeline_step(drafter: int, latents, n: int, text_ctx, draft_schedule, skip_mask,
                     proxy_plan, refiner=None, refine_latent=None, refine_schedule=None,
                     draft_opts=None, refine_opts=None) -> None:
    """Drafts `latents` with `drafter` while `refiner` refines `refine_latent` (the
    previous pool's selected candidate) on a worker thread of the library; returns when
    both are done. refine_latent None: the draft alone."""
    ds = np.ascontiguousarray(draft_schedule, np.float32)
    sk = None if skip_mask is None else np.ascontiguousarray(skip_mask, np.uint8)
    px = None if proxy_plan is None else np.ascontiguousarray(proxy_plan, np.int32)
    rsched = (np.zeros(1, np.float32) if refine_schedule is None
              else np.ascontiguousarray(refine_schedule, np.float32))
    _check(load_library().fb_pipeline_step(
        drafter, _ptr(latents, np.float32), n, _ptr(text_ctx, np.float32), _ptr(ds),
        len(ds) - 1, _ptr(sk), _ptr(px), None if draft_opts is None else ctypes.byref(draft_opts),
        refiner, _ptr(refine_latent, np.float32), _ptr(rsched), len(rsched) - 1,
        None if refine_opts is None else ctypes.byref(refine_opts)))


def fb_select_elo(scores, compare, rho1=0.5, rho2=0.5, kappa=1.5, k_base=32.0):
    """Stage 2 selection. compare(a, b) -> (a_preferred, confidence 0/1/2).
    Returns (winner, ratings [M], pairwise calls)."""
    sc = np.ascontiguousarray(scores, np.int32)
    M = sc.size

    def cb(user, a, b, conf_ptr):
        pref, conf = compare(a, b)
        conf_ptr[0] = int(conf)
        return 1 if pref else 0
    fn = PAIR_VERIFIER(cb)
    winner, calls = ctypes.c_int(), ctypes.c_int()
    ratings = np.zeros(M, np.float64)
    _check(load_library().fb_select_elo(_ptr(sc), M, rho1, rho2, kappa, k_base, fn, None,
                                        ctypes.byref(winner),
                                        ratings.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                                        ctypes.byref(calls)))
    return winner.value, ratings, calls.value


def fb_plan_from_phi(S, S_prime, n_skip, l_start, l_end, f_full, order, depth):
    skip = np.zeros((S_prime, depth), np.uint8)
    proxy = np.zeros((S_prime, depth), np.int32)
    _check(load_library().fb_plan_from_phi(S, S_prime, n_skip, l_start, l_end, f_full, order,
                                           depth, _ptr(skip), _ptr(proxy)))
    return skip, proxy


def fb_block_forward(model: int, layer: int, h, n: int, t: float) -> None:
    _check(load_library().fb_block_forward(model, layer, _ptr(h), n, float(t)))


def fb_set_timing(model: int, mask: int) -> None:
    _check(load_library().fb_set_timing(model, int(mask)))


def fb_set_op_repeat(model: int, n: int) -> None:
    _check(load_library().fb_set_op_repeat(model, int(n)))


def fb_set_device_wait_limit(ns: int) -> None:
    """Device-side wait limit in nanoseconds (0 = the default 2 s); a testing hook."""
    _check(load_library().fb_set_device_wait_limit(int(ns)))


def fb_test_fail_alloc(k: int) -> None:
    """Makes the library's k-th device allocation from now fail (k < 0 disarms)."""
    _check(load_library().fb_test_fail_alloc(int(k)))


def fb_test_alloc_calls() -> int:
    """Device allocations the library made since the last fb_test_fail_alloc."""
    return int(load_library().fb_test_alloc_calls())


def fb_test_poison_counters(model) -> None:
    """Sets the stream-K counters of `model` (None: the allocation-free entry point's) to
    a large negative value, so the next stream-K finisher's wait cannot complete."""
    _check(load_library().fb_test_poison_counters(model))


def fb_probe_mma_rate(issuers: int, n: int, reps: int = 16384) -> float:
    """Tensor-pipe MACs per SM clock with `issuers` issuing warps and M=128 x n MMAs."""
    out = ctypes.c_double()
    _check(load_library().fb_probe_mma_rate(int(issuers), int(n), int(reps), ctypes.byref(out)))
    return out.value


def fb_probe_mma_gap(gap: int) -> float:
    """Tensor-pipe MACs per SM clock with a gap of `gap` clocks after every 8 MMAs."""
    out = ctypes.c_double()
    _check(load_library().fb_probe_mma_gap(int(gap), ctypes.byref(out)))
    return out.value


def fb_probe_mufu(op: int) -> float:
    """Results per SM clock of ex2 (0), tanh (1), rcp (2) or ex2 on f16 pairs (3)."""
    out = ctypes.c_double()
    _check(load_library().fb_probe_mufu(int(op), ctypes.byref(out)))
    return out.value


def fb_probe_tmem_load(busy: bool) -> float:
    """SM clocks of a 128-column TMEM load and its wait (tensor pipe idle or running)."""
    out = ctypes.c_double()
    _check(load_library().fb_probe_tmem_load(1 if busy else 0, ctypes.byref(out)))
    return out.value


def fb_probe_mma_mix(form: int, loaders: int = 0, loader_gap: int = 0) -> float:
    """Tensor-pipe MACs per SM clock of attention-step-shaped MMA batches (form 0: both
    operands K-major in shared memory, 1: B MN-major, 2: B MN-major and A from TMEM, 3: a
    whole attention step, 4: the same with its commits, 5 and 6: forms 3 and 4 with hoisted
    descriptor words; 7-13: forms 0-6 with softmax arithmetic in the loaders) with `loaders`
    warps reading and writing TMEM meanwhile."""
    out = ctypes.c_double()
    _check(load_library().fb_probe_mma_mix(int(form), int(loaders), int(loader_gap),
                                           ctypes.byref(out)))
    return out.value


def fb_get_stats(model: int) -> dict:
    arr = (fb_kstat * len(KERNEL_KINDS))()
    _check(load_library().fb_get_stats(model, ctypes.cast(arr, ctypes.c_void_p)))
    return {KERNEL_KINDS[i]: dict(launches=int(arr[i].launches), ms=arr[i].ms,
                                  flops=arr[i].flops, bytes=arr[i].bytes)
            for i in range(len(KERNEL_KINDS))}


def fb_reset_stats(model: int) -> None:
    _check(load_library().fb_reset_stats(model))


def fb_op_gemm(model, M, N, K, A, W, bias, epi, out, resid=None, gate=None, base=None,
               delta=None, impl=0) -> None:
    _check(load_library().fb_op_gemm(model, M, N, K, _ptr(A), _ptr(W), _ptr(bias), epi,
                                     _ptr(out), _ptr(resid), _ptr(gate), _ptr(base),
                                     _ptr(delta), impl))


def fb_gemm_streamk_noalloc(stream, M, N, K, A, W, bias, epi, out, resid=None, gate=None,
                            base=None, delta=None) -> None:
    """The allocation-free stream-K GEMM (no model); `stream` is a cudaStream_t handle
    (int) or None for the legacy default stream. Waits for the result."""
    _check(load_library().fb_gemm_streamk_noalloc(stream, M, N, K, _ptr(A), _ptr(W),
                                                  _ptr(bias), epi, _ptr(out), _ptr(resid),
                                                  _ptr(gate), _ptr(base), _ptr(delta)))


def fb_op_attention(model, Q, ldq, Kt, ldk, V, ldv, O, ldo, batch, Lq, Lkv, kv_batch_rows,
                    heads, head_dim, impl=0) -> None:
    _check(load_library().fb_op_attention(model, _ptr(Q), ldq, _ptr(Kt), ldk, _ptr(V), ldv,
                                          _ptr(O), ldo, batch, Lq, Lkv, kv_batch_rows, heads,
                                          head_dim, impl))


class Model:
    """Owns an fb_model handle; methods forward to the fb_* functions."""

    def __init__(self, cfg: synth.Cfg, weights):
        self.cfg = cfg
        self.handle = fb_init_model(cfg, weights)

    def close(self):
        if self.handle:
            fb_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def set_stream(self, stream):
        fb_set_stream(self.handle, stream)

    def set_sm_budget(self, n_sms):
        fb_set_sm_budget(self.handle, n_sms)

    def encode_text(self, ctx):
        fb_encode_text(self.handle, ctx)

    def draft(self, latents, text_ctx, schedule, skip_mask=None, proxy_plan=None, n=None,
              opts=None):
        n = latents.shape[0] if n is None else n
        if opts is None:
            fb_draft(self.handle, latents, n, text_ctx, schedule, skip_mask, proxy_plan)
        else:
            fb_draft_ex(self.handle, latents, n, text_ctx, schedule, skip_mask, proxy_plan, opts)

    def refine(self, latent, text_ctx, schedule, opts=None):
        if opts is None:
            fb_refine(self.handle, latent, text_ctx, schedule)
        else:
            fb_refine_ex(self.handle, latent, text_ctx, schedule, opts)

    def state_bytes(self) -> int:
        return fb_state_bytes(self.handle)

    def state_offload(self, first, dsts):
        fb_state_offload(self.handle, first, dsts)

    def state_wait(self):
        fb_state_wait(self.handle)

    def block_forward(self, layer, h, n, t):
        fb_block_forward(self.handle, layer, h, n, t)

    def set_timing(self, mask):
        fb_set_timing(self.handle, mask)

    def stats(self):
        return fb_get_stats(self.handle)

    def reset_stats(self):
        fb_reset_stats(self.handle)
