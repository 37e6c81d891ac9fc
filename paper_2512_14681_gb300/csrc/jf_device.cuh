// Device-side helpers of libjf: inline PTX for sm_103a (mbarrier, TMA, tcgen05, programmatic
// dependent launch), bounded waits and the shared error flag.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "jf_internal.h"

#define JF_DEV __device__ __forceinline__

typedef __nv_bfloat16 bf16;


JF_DEV void jf_set_error(int* err, int code) {
  if (err) atomicCAS(err, 0, code);
}

JF_DEV uint64_t jf_globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Kernel ids of the timeline records.
enum TlKernel : unsigned {
  TL_NORM = 1, TL_NORM_ACC = 2, TL_QKV_FINISH = 3, TL_ATTN = 5, TL_GEMM = 10 /* + epilogue kind */,
  TL_EMBED = 20, TL_ACCEPT = 21, TL_COMMIT = 22
};

// Timeline of the forward's kernels, compiled in only with -DJF_TIMELINE (the default build has
// none of it): thread 0 of every CTA records its kernel id, block, SM, entry time, the time it got
// past its dependency wait and its exit time, into a caller buffer set by jf_tl_enable().
#ifdef JF_TIMELINE
struct TlRec {
  unsigned kid, blk, smid, pad;
  unsigned long long t0, t1, t2;
};
constexpr int kTlMaxRecords = 2000000;
static __device__ TlRec* jf_tl_buf;  // one pair per translation unit, set by its own setter
static __device__ int* jf_tl_idx;
JF_DEV void jf_tl_record(unsigned kid, uint64_t t0, uint64_t t1) {
  if (!jf_tl_buf) return;
  const uint64_t t2 = jf_globaltimer();
  unsigned sm;
  asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
  const int i = atomicAdd(jf_tl_idx, 1);
  if (i < kTlMaxRecords) jf_tl_buf[i] = TlRec{kid, blockIdx.x, sm, 0u, t0, t1, t2};
}
#define JF_TL_ENTRY()                       \
  const uint64_t jf_tl_t0 = jf_globaltimer(); \
  uint64_t jf_tl_t1 = 0
#define JF_TL_WAITED() (jf_tl_t1 = jf_globaltimer())
#define JF_TL_EXIT(kid)                                               \
  do {                                                                \
    if (threadIdx.x == 0) jf_tl_record((unsigned)(kid), jf_tl_t0, jf_tl_t1); \
  } while (0)
#define JF_TL_SETTER(name)                                                     \
  cudaError_t name(void* records, void* counter) {                             \
    cudaError_t e = cudaMemcpyToSymbol(jf_tl_buf, &records, sizeof(void*));   \
    return e != cudaSuccess ? e : cudaMemcpyToSymbol(jf_tl_idx, &counter, sizeof(void*)); \
  }
#else
#define JF_TL_ENTRY() \
  do {                \
  } while (0)
#define JF_TL_WAITED() \
  do {                 \
  } while (0)
#define JF_TL_EXIT(kid) \
  do {                  \
  } while (0)
#endif

// ------------------------------------------------------------------------------------------
// Programmatic dependent launch. Every kernel of the chain calls pdl_wait() before it reads
// anything an earlier kernel wrote (and before it exits), so completion stays transitive.
// ------------------------------------------------------------------------------------------
JF_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
JF_DEV void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ------------------------------------------------------------------------------------------
// Shared-memory addresses, mbarriers
// ------------------------------------------------------------------------------------------
JF_DEV uint32_t smem_u32(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }

JF_DEV void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

JF_DEV void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }

JF_DEV void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

JF_DEV void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

JF_DEV bool mbar_try_wait(uint32_t bar, uint32_t parity) {
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

// Wait for phase `parity` of an mbarrier, giving up after `limit_ns` nanoseconds.
JF_DEV bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = jf_globaltimer();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (jf_globaltimer() - t0 > limit_ns) return false;
  }
}


// ------------------------------------------------------------------------------------------
// Thread-block clusters: ranks, cluster-wide barrier
// ------------------------------------------------------------------------------------------
JF_DEV uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
JF_DEV uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
JF_DEV void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// ------------------------------------------------------------------------------------------
// TMA (cp.async.bulk.tensor) loads with an L2 cache-policy hint
// ------------------------------------------------------------------------------------------
JF_DEV uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

JF_DEV uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// 2-D tiled load: box at coordinates (c0 = innermost, c1) into shared memory, completing
// `bytes` on mbarrier `bar`. The innermost coordinate is always a multiple of 64 elements
// (128 bytes) here, which keeps every copy on a 16-byte boundary.
JF_DEV void tma_load_2d(uint32_t smem_dst, const void* tmap, uint32_t bar, int c0, int c1, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_dst),
      "l"(tmap), "r"(c0), "r"(c1), "r"(bar), "l"(policy)
      : "memory");
}

JF_DEV void tma_prefetch_desc(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(tmap) : "memory");
}

// ------------------------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, accumulator in tensor memory)
// ------------------------------------------------------------------------------------------
JF_DEV void tmem_alloc(uint32_t smem_result, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_result), "r"(ncols)
               : "memory");
}
JF_DEV void tmem_relinquish() { asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory"); }
JF_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
JF_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
JF_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulate), one CTA.
JF_DEV void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on an mbarrier when all previously issued tcgen05 MMAs of this thread complete.
JF_DEV void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// Load 16 consecutive fp32 columns of this warp's 32 TMEM lanes (lane = thread).
JF_DEV void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Load 32 consecutive fp32 columns of this warp's 32 TMEM lanes (lane = thread).
JF_DEV void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor for a K-major operand tile written by TMA with 128-byte
// swizzle: rows of 128 bytes, 8-row swizzle atoms 1024 bytes apart (stride byte offset),
// descriptor version 1, layout type 2 (SWIZZLE_128B).
JF_DEV uint64_t sdesc_k_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)(16u >> 4) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Shared-memory descriptor of an MN-major operand with the 128-byte swizzle: rows of 64 MN
// elements (128 bytes) at consecutive K indices, swizzled in 8-row groups 1024 bytes apart (stride
// byte offset); consecutive 64-element MN atoms `lbo` bytes apart (leading byte offset).
JF_DEV uint64_t sdesc_mn_sw128(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
// The same with fp16 A and B (A and B of one MMA always share their type).
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ------------------------------------------------------------------------------------------
// Small numeric helpers
// ------------------------------------------------------------------------------------------
template <typename T>
JF_DEV T to_act(float v);
template <>
JF_DEV float to_act<float>(float v) { return v; }
template <>
JF_DEV bf16 to_act<bf16>(float v) { return __float2bfloat16_rn(v); }

JF_DEV float act_to_f32(float v) { return v; }
JF_DEV float act_to_f32(bf16 v) { return __bfloat162float(v); }

JF_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

JF_DEV float silu_f(float x) { return x / (1.0f + __expf(-x)); }

// (value, index) ordering of the greedy decision: larger value wins, lower index on ties.
JF_DEV bool better(float v, int i, float bv, int bi) { return v > bv || (v == bv && i < bi); }
