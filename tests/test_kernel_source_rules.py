"""Static checks on the CUDA sources (no GPU needed)."""
import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2607_04461_gb300", "csrc")


def kernels():
    for f in sorted(os.listdir(CSRC)):
        if not f.endswith(".cu"):
            continue
        src = open(os.path.join(CSRC, f)).read()
        for m in re.finditer(r"__global__[^{;]*?\b(\w+)\s*\(", src, flags=re.S):
            # body: from the first "{" after the signature to its matching "}"
            i = src.index("{", m.end())
            depth, j = 0, i
            while True:
                if src[j] == "{":
                    depth += 1
                elif src[j] == "}":
                    depth -= 1
                    if depth == 0:
                        break
                j += 1
            yield f, m.group(1), src[i:j]


def test_every_kernel_waits_for_its_predecessor():
    """Kernels are launched with programmatic stream serialisation, so each must call
    griddep_wait() before it reads what the previous kernel wrote."""
    found = list(kernels())
    assert len(found) >= 15
    missing = [f"{f}:{name}" for f, name, body in found if "griddep_wait()" not in body]
    assert not missing, missing


def test_every_kernel_is_launched_through_launch_k():
    for f in os.listdir(CSRC):
        if f.endswith(".cu"):
            assert "<<<" not in open(os.path.join(CSRC, f)).read(), f


def _function_body(src, name):
    i = src.index("{", src.index(name + "("))
    depth, j = 0, i
    while True:
        if src[j] == "{":
            depth += 1
        elif src[j] == "}":
            depth -= 1
            if depth == 0:
                return src[i:j]
        j += 1


def test_noalloc_entry_point_allocates_nothing():
    """fb_gemm_streamk_noalloc and its set-up use static device arrays only: no
    allocating call anywhere on their path."""
    src = open(os.path.join(CSRC, "api.cu")).read()
    body = _function_body(src, "fb_status fb_gemm_streamk_noalloc") + \
        _function_body(src, "fb_status noalloc_setup")
    for bad in ("Malloc", "Free", "dalloc", "new ", "std::vector", "cudaMemPool"):
        assert bad not in body, bad
    assert body.count("cudaGetSymbolAddress") == 3
    assert re.search(r"static __device__ __align__\(256\) float g_na_ws\[", src)
