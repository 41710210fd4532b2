// Device helpers shared by the sm_103a kernels of the draft path.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

typedef __nv_bfloat16 bf16;

// Error codes a kernel writes to the model's device error word.
enum { FB_DEVERR_NONE = 0, FB_DEVERR_WAIT_TIMEOUT = 1, FB_DEVERR_BAD_ARG = 2 };

// Time limit of one device-side wait (ns); a wait that runs past it reports
// FB_DEVERR_WAIT_TIMEOUT and makes the kernel give up. Each translation unit that waits
// holds its own copy of the limit (no relocatable device code); fb_set_wait_limit_tu
// sets the copy of the calling unit on the current device.
#define FB_WAIT_LIMIT_NS 2000000000ull
static __device__ unsigned long long g_fb_wait_limit_ns = FB_WAIT_LIMIT_NS;
__device__ __forceinline__ unsigned long long fb_wait_limit() {
  return *(volatile unsigned long long*)&g_fb_wait_limit_ns;
}
static inline cudaError_t fb_set_wait_limit_tu(unsigned long long ns) {
  return cudaMemcpyToSymbol(g_fb_wait_limit_ns, &ns, sizeof(ns));
}

__device__ __forceinline__ uint64_t fb_globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---- programmatic dependent launch ---------------------------------------------------
// Kernels of the path are launched with programmatic stream serialisation: a kernel may
// be scheduled while its predecessor on the stream is still running, runs its prologue
// (barrier init, TMEM allocation, descriptor prefetch), and waits in griddep_wait() until
// the predecessor has completed and its writes are visible. griddep_launch() lets the
// successor be scheduled (it only starts once every CTA of this grid has called it or
// exited). Both are no-ops for a kernel launched without the attribute.
__device__ __forceinline__ void griddep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void griddep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

#ifdef __CUDACC__
// The programmatic relaxation only orders a kernel after a preceding KERNEL that calls
// griddepcontrol; a copy, memset or event record before it gives no such ordering. So
// the attribute is used only when the previous operation this host thread put on the
// stream was one of these kernels: every other stream operation of the library calls
// fb_stream_op_not_kernel(). FB_NO_PDL in the environment (read once) disables it.
bool fb_pdl_enabled();
bool fb_prev_op_is_kernel();
void fb_set_prev_op_is_kernel(bool v);
inline void fb_stream_op_not_kernel() { fb_set_prev_op_is_kernel(false); }
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = (fb_pdl_enabled() && fb_prev_op_is_kernel()) ? 1 : 0;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
  fb_set_prev_op_is_kernel(e == cudaSuccess);
  return e;
}
#endif

// ---- bf16 packing --------------------------------------------------------------
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_bf16x2(uint32_t u) {
  __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
  return __bfloat1622float2(v);
}
__device__ __forceinline__ void load_bf16x8(const bf16* p, float* v) {
  uint4 u = *reinterpret_cast<const uint4*>(p);
  float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y), c = unpack_bf16x2(u.z),
         d = unpack_bf16x2(u.w);
  v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
  v[4] = c.x; v[5] = c.y; v[6] = d.x; v[7] = d.y;
}
__device__ __forceinline__ void store_bf16x8(bf16* p, const float* v) {
  uint4 u;
  u.x = pack_bf16x2(v[0], v[1]); u.y = pack_bf16x2(v[2], v[3]);
  u.z = pack_bf16x2(v[4], v[5]); u.w = pack_bf16x2(v[6], v[7]);
  *reinterpret_cast<uint4*>(p) = u;
}
// one 32-byte store (p 32-byte aligned)
__device__ __forceinline__ void store_b32x8(void* p, const uint32_t* w) {
  asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(w[0]), "r"(w[1]),
               "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
               : "memory");
}
__device__ __forceinline__ void load_f32x8(const float* p, float* v) {
  float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void store_f32x8(float* p, const float* v) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}

__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// GELU, tanh form: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3))), evaluated as
// h + h tanh(x (k0 + k1 x^2)) with h = x / 2 (five fp32 operations and one tanh). The
// hardware tanh (max relative error about 2^-11) is well inside the bf16 rounding of the
// GEMM output that it feeds.
__device__ __forceinline__ float gelu_tanh_f(float x) {
  const float k0 = 0.7978845608028654f;              // sqrt(2/pi)
  const float k1 = 0.7978845608028654f * 0.044715f;  // sqrt(2/pi) * 0.044715
  const float h = 0.5f * x;
  return fmaf(h, tanh_approx(x * fmaf(x * x, k1, k0)), h);
}
// packed pairs of fp32 (sm_100 and later execute one fma/add/mul on both halves)
__device__ __forceinline__ uint64_t f2_join(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
// gelu_tanh_f on a pair, the fp32 arithmetic on packed pairs
__device__ __forceinline__ void gelu_tanh_f2(float& a, float& b) {
  const uint64_t x = f2_join(a, b);
  const uint64_t h = f2_mul(x, f2_join(0.5f, 0.5f));
  const uint64_t t = f2_fma(f2_mul(x, x), f2_join(0.7978845608028654f * 0.044715f,
                                                   0.7978845608028654f * 0.044715f),
                            f2_join(0.7978845608028654f, 0.7978845608028654f));
  float u0, u1;
  f2_split(f2_mul(x, t), u0, u1);
  const uint64_t th = f2_join(tanh_approx(u0), tanh_approx(u1));
  f2_split(f2_fma(h, th, h), a, b);
}
__device__ __forceinline__ float silu_f(float x) { return x / (1.f + expf(-x)); }

// ---- mbarrier ------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Waits until the phase with the given parity has completed. Gives up after
// FB_WAIT_LIMIT_NS (or at once if another role already reported an error), records
// the timeout in *err and returns false.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* err) {
  const uint32_t a = smem_u32(bar);
  if (mbar_try(a, parity)) return true;
  const uint64_t t0 = fb_globaltimer();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try(a, parity)) return true;
    if ((i & 63u) == 0) {
      if (*(volatile int*)err != 0) return false;
      if (fb_globaltimer() - t0 > fb_wait_limit()) {
        atomicExch(err, FB_DEVERR_WAIT_TIMEOUT);
        return false;
      }
    }
  }
}

// ---- TMA -----------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}
// Untiled bulk copy global -> shared (both 16-byte aligned, bytes a multiple of 16),
// completing on an mbarrier like the tiled loads.
__device__ __forceinline__ void bulk_load_1d(void* dst, const void* src, uint32_t bytes,
                                             uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
// Orders this thread's earlier generic-proxy accesses to global memory (and what they
// observed) before its later async-proxy (bulk copy) accesses.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
// TMA store of a shared-memory tile (bulk async-group completion)
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];"
               ::"l"(reinterpret_cast<uint64_t>(map)), "r"(src), "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// at most N committed bulk groups still reading their shared-memory source
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// at most N committed bulk groups not yet complete
template <int N>
__device__ __forceinline__ void bulk_wait() {
  asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}
// generic-proxy shared-memory writes become visible to the async proxy (TMA)
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---- tcgen05 (5th-generation tensor core, accumulators in tensor memory) -------
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Whole warp: allocates ncols TMEM columns, writes the base address to *holder (smem).
__device__ __forceinline__ void tmem_alloc(uint32_t* holder, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(holder)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulate).
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrives once on *bar when all tcgen05.mma issued so far by this thread are done.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
// 32 lanes x 32 consecutive 32-bit columns: thread i gets lane (taddr.lane + i).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// Emits nothing; makes 32 registers filled by tcgen05.ld look written at this point, so
// no use of them is scheduled before the tcgen05.wait::ld that precedes it.
__device__ __forceinline__ void reg_fence32(uint32_t* r) {
  asm volatile(""
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]),
                 "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
                 "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]),
                 "+r"(r[30]), "+r"(r[31]));
}

// Shared-memory matrix descriptors with 128-byte swizzle, split into their two 32-bit
// words. The upper word (stride byte offset 1024 B, version bit, 128-byte swizzle) is one
// constant; the lower word holds the start address >> 4 (bits 0-13) and the leading byte
// offset >> 4 (bits 16-29), so the
// descriptor of an operand slice `off` bytes further on is lower word + (off >> 4) (shared
// addresses stay below 256 KB: the start field cannot carry into the offset field).
constexpr uint32_t DESC_HI = (1024u >> 4) | (1u << 14) | (2u << 29);
__device__ __forceinline__ uint32_t desc_lo_k(uint32_t saddr) {
  return ((saddr & 0x3FFFFu) >> 4) | (1u << 16);
}
__device__ __forceinline__ uint32_t desc_lo_mn(uint32_t saddr, uint32_t lbo) {
  return ((saddr & 0x3FFFFu) >> 4) | (((lbo >> 4) & 0x3FFFu) << 16);
}
// tcgen05.mma kind::f16 from the descriptors' lower words (A and B in shared memory, or A
// in TMEM): the issuing thread spends one add per operand and instruction, which keeps it
// ahead of the tensor pipe while softmax warps share its SM sub-partition
__device__ __forceinline__ void tc_mma_ss_lo(uint32_t d_tmem, uint32_t alo, uint32_t blo,
                                             uint32_t hi, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 da, db;\n\t"
      "setp.ne.b32 p, %5, 0;\n\t"
      "mov.b64 da, {%1, %3};\n\t"
      "mov.b64 db, {%2, %3};\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], da, db, %4, p;\n\t}" ::"r"(d_tmem),
      "r"(alo), "r"(blo), "r"(hi), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_mma_ts_lo(uint32_t d_tmem, uint32_t a_tmem, uint32_t blo,
                                             uint32_t hi, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 db;\n\t"
      "setp.ne.b32 p, %5, 0;\n\t"
      "mov.b64 db, {%2, %3};\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], db, %4, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "r"(blo), "r"(hi), "r"(idesc), "r"(accumulate)
      : "memory");
}

// ---- clusters and the 2-SM (cta_group::2) forms -----------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// All threads of all CTAs of the cluster (release / acquire).
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}
// shared::cluster address of the same shared-memory location in CTA `rank`.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}
// TMA tile load into this CTA's shared memory whose completion is signalled on an
// mbarrier that may live in the peer CTA of the pair (shared::cluster address).
__device__ __forceinline__ void tma_load_2d_cg2(void* dst, const CUtensorMap* map,
                                                uint32_t mbar_cluster, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(mbar_cluster)
      : "memory");
}
// Pair-wide TMEM allocation: one warp in each CTA of the pair executes it.
__device__ __forceinline__ void tmem_alloc_cg2(uint32_t* holder, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(holder)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_cg2(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// D[tmem of both CTAs] (+)= A[smem of both CTAs, 128 rows each] * B^T[smem, N/2 rows each].
__device__ __forceinline__ void tc_mma_f16_cg2(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                               uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrives once on the mbarrier at this shared-memory offset in every CTA of cta_mask
// when all tcgen05.mma issued so far by this thread are done.
__device__ __forceinline__ void tc_commit_mc(uint64_t* bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(cta_mask)
      : "memory");
}

// Bulk prefetch of [p, p + bytes) into L2 (p and bytes multiples of 16).
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(p)),
               "r"(bytes)
               : "memory");
}

// ---- GEMM epilogue (shared by the tcgen05 and CUDA-core GEMMs) --------------------
enum { EPI_BF16 = 0, EPI_GELU_BF16 = 1, EPI_RESID = 2, EPI_RESID_DELTA = 3 };

// stream-K state passed to the 2-SM GEMM kernel (see its work-split comment)
struct SkArgs {
  int on;
  float* ws;
  int* ctr;
};

struct GemmEpi {
  const float* bias;   // [N] or null
  void* out;           // bf16 (EPI_BF16, EPI_GELU_BF16) or fp32 (EPI_RESID*)
  const float* resid;  // fp32 [M][ldo]; EPI_RESID: null = no residual (out = gate * (acc + bias))
  const float* gate;   // fp32 [N] or null (= 1)
  const float* base;   // fp32 [M][ldo] (EPI_RESID_DELTA)
  bf16* delta;         // bf16 [M][ldo] (EPI_RESID_DELTA)
  int ldo;
};

// Residual epilogues read fp32 rows from HBM; the epilogue warps prefetch their part of
// the next tile's rows into L2 while the mainloop runs, so those reads hit L2.
template <int KIND>
__device__ __forceinline__ void epi_prefetch(const GemmEpi& e, int row, int col, int ncols) {
  if (KIND >= EPI_RESID && e.resid) {
    const size_t off = (size_t)row * e.ldo + col;
    prefetch_l2_bulk(e.resid + off, ncols * 4);
    if (KIND == EPI_RESID_DELTA && e.base != e.resid) prefetch_l2_bulk(e.base + off, ncols * 4);
  }
}

// Applies the epilogue to 32 consecutive accumulators v of row `row`, columns
// col..col+31. Every global load of the chunk is issued before its first store (out may
// alias resid / base element for element, so this order is safe), which keeps 32 B x 12
// loads in flight per thread instead of serialising load -> store per 8 columns.
template <int KIND>
__device__ __forceinline__ void epi_apply32(const GemmEpi& e, int row, int col, float* v) {
  const size_t off = (size_t)row * e.ldo + col;
  if (KIND >= EPI_RESID) {
    // the row-dependent operands (HBM) first; gate and bias are the same for every row
    // (L1-resident) and are read per 8 columns while computing
    float r[32], bs[32];
#pragma unroll
    for (int j = 0; j < 32; j += 8) {
      if (KIND == EPI_RESID_DELTA || e.resid) {
        load_f32x8(e.resid + off + j, r + j);
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) r[j + q] = 0.f;
      }
      if (KIND == EPI_RESID_DELTA) load_f32x8(e.base + off + j, bs + j);
    }
#pragma unroll
    for (int j = 0; j < 32; j += 8) {
      float g[8], b[8];
      if (e.gate) load_f32x8(e.gate + col + j, g);
      if (e.bias) load_f32x8(e.bias + col + j, b);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float a = v[j + q] + (e.bias ? b[q] : 0.f);
        v[j + q] = r[j + q] + (e.gate ? g[q] : 1.f) * a;
      }
    }
    if (KIND == EPI_RESID_DELTA) {
#pragma unroll
      for (int j = 0; j < 32; j += 8) {
        float d[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) d[q] = v[j + q] - bs[j + q];
        store_bf16x8(e.delta + off + j, d);
      }
    }
#pragma unroll
    for (int j = 0; j < 32; j += 8) store_f32x8(reinterpret_cast<float*>(e.out) + off + j, v + j);
  } else {
    if (e.bias) {
      float b[32];
#pragma unroll
      for (int j = 0; j < 32; j += 8) load_f32x8(e.bias + col + j, b + j);
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] += b[j];
    }
    if (KIND == EPI_GELU_BF16) {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = gelu_tanh_f(v[j]);
    }
#pragma unroll
    for (int j = 0; j < 32; j += 8) store_bf16x8(reinterpret_cast<bf16*>(e.out) + off + j, v + j);
  }
}

// Applies the epilogue to 8 consecutive accumulators v of row `row`, columns col..col+7.
template <int KIND>
__device__ __forceinline__ void epi_apply8(const GemmEpi& e, int row, int col, float* v) {
  if (e.bias) {
    float b[8];
    load_f32x8(e.bias + col, b);
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] += b[j];
  }
  const size_t off = (size_t)row * e.ldo + col;
  if (KIND == EPI_BF16) {
    store_bf16x8(reinterpret_cast<bf16*>(e.out) + off, v);
  } else if (KIND == EPI_GELU_BF16) {
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = gelu_tanh_f(v[j]);
    store_bf16x8(reinterpret_cast<bf16*>(e.out) + off, v);
  } else {
    float r[8], g[8];
    if (KIND == EPI_RESID_DELTA || e.resid) {
      load_f32x8(e.resid + off, r);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) r[j] = 0.f;
    }
    if (e.gate) {
      load_f32x8(e.gate + col, g);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) g[j] = 1.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = r[j] + g[j] * v[j];
    if (KIND == EPI_RESID_DELTA) {
      float b[8], d[8];
      load_f32x8(e.base + off, b);
#pragma unroll
      for (int j = 0; j < 8; ++j) d[j] = v[j] - b[j];
      store_bf16x8(e.delta + off, d);
    }
    store_f32x8(reinterpret_cast<float*>(e.out) + off, v);
  }
}
