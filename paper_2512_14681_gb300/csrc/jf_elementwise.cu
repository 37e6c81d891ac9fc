// Small kernels of the forward pass: random weights, the rotary table, embedding lookup and
// RMSNorm (the Qwen2.5-style decoder of Sec. 4.1).
#include "jf_device.cuh"
#include "jf_internal.h"

namespace jf {
namespace {

// SplitMix64 (Steele, Lea & Flood 2014): the i-th output of a stream started at state s.
__device__ __forceinline__ uint64_t sm64_out(uint64_t s, uint64_t i) {
  uint64_t z = s + (i + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Weight tensor of `rows` x `cols` logical entries, entry e = std * N(0,1) drawn by Box-Muller
// from outputs 2j, 2j+1 (j = e / 2) of the SplitMix64 stream keyed by output `tid` of the stream
// seeded with `seed`. Logical row r lands at device row (r / grp) * grp_stride + r % grp + grp_off.
template <typename T>
__global__ void k_init_weights(T* dst, long long rows, long long cols, uint64_t seed, uint64_t tid, double stdv,
                               long long grp, long long grp_stride, long long grp_off) {
  const long long n = rows * cols;
  const long long npairs = (n + 1) / 2;
  const uint64_t s = sm64_out(seed, tid);
  const double two53 = 9007199254740992.0;
  for (long long j = blockIdx.x * (long long)blockDim.x + threadIdx.x; j < npairs;
       j += (long long)gridDim.x * blockDim.x) {
    const uint64_t a = sm64_out(s, 2ull * j), b = sm64_out(s, 2ull * j + 1);
    const double u1 = ((double)(a >> 11) + 1.0) / two53;
    const double u2 = (double)(b >> 11) / two53;
    const double rad = sqrt(-2.0 * log(u1));
    double sn, cs;
    sincos(2.0 * 3.14159265358979323846 * u2, &sn, &cs);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const long long e = 2 * j + h;
      if (e >= n) break;
      const double z = stdv * rad * (h ? sn : cs);
      const long long r = e / cols, c = e % cols;
      const long long dr = (r / grp) * grp_stride + (r % grp) + grp_off;
      if constexpr (sizeof(T) == 2) dst[dr * cols + c] = __double2bfloat16(z);
      else dst[dr * cols + c] = (float)z;
    }
  }
}

__global__ void k_fill_f32(float* p, long long n, float v) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
    p[i] = v;
}

// (cos, sin) of position * theta^(-2i/hd), computed in fp64 and stored as fp32.
__global__ void k_rope_table(float2* tab, int n_pos, int half, double theta) {
  const long long n = (long long)n_pos * half;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n; e += (long long)gridDim.x * blockDim.x) {
    const int p = (int)(e / half), i = (int)(e % half);
    const double inv = pow(theta, -(2.0 * i) / (2.0 * half));
    double sn, cs;
    sincos((double)p * inv, &sn, &cs);
    tab[e] = make_float2((float)cs, (float)sn);
  }
}

// x[r, :] = E[tok[r], :] (fp32 residual stream)
template <typename T>
__global__ void k_embed(const T* __restrict__ E, const int* __restrict__ tok, float* __restrict__ x, int d, int V,
                        int* err) {
  JF_TL_ENTRY();
  pdl_launch_dependents();
  pdl_wait();
  JF_TL_WAITED();
  const int r = blockIdx.x;
  int t = tok[r];
  if (t < 0 || t >= V) {
    if (threadIdx.x == 0) jf_set_error(err, JF_DERR_BOUNDS);
    t = 0;
  }
  // 16-byte vectors (d is a multiple of 64, so every row starts 128-byte aligned); up to four
  // vectors a thread are loaded before the first store, so a row costs one round trip to memory
  constexpr int VE = 16 / sizeof(T);  // elements per vector
  const uint4* src = reinterpret_cast<const uint4*>(E + (size_t)t * d);
  float4* dst = reinterpret_cast<float4*>(x + (size_t)r * d);
  const int nv = d / VE;
  for (int base = 0; base < nv; base += 4 * (int)blockDim.x) {
    uint4 w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int i = base + k * (int)blockDim.x + (int)threadIdx.x;
      w[k] = (i < nv) ? src[i] : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int i = base + k * (int)blockDim.x + (int)threadIdx.x;
      if (i >= nv) continue;
      if constexpr (VE == 8) {  // bf16: 8 values -> two float4
        dst[2 * i] = make_float4(__uint_as_float(w[k].x << 16), __uint_as_float(w[k].x & 0xffff0000u),
                                 __uint_as_float(w[k].y << 16), __uint_as_float(w[k].y & 0xffff0000u));
        dst[2 * i + 1] = make_float4(__uint_as_float(w[k].z << 16), __uint_as_float(w[k].z & 0xffff0000u),
                                     __uint_as_float(w[k].w << 16), __uint_as_float(w[k].w & 0xffff0000u));
      } else {  // fp32: 4 values
        dst[i] = make_float4(__uint_as_float(w[k].x), __uint_as_float(w[k].y), __uint_as_float(w[k].z),
                             __uint_as_float(w[k].w));
      }
    }
  }
  JF_TL_EXIT(TL_EMBED);
}

// y[r, :] = x[r, :] / sqrt(mean(x[r, :]^2) + eps) * gain, rounded to the activation type.
// One CTA of 1024 threads per row; the row stays in registers (float4, up to 2 per thread:
// d <= 8192), so x is read once. The reduction order is fixed by d alone.
// ACC: the residual update of the preceding projection is finished here first: the k_splits
// partial sums of x's increment (EPI_PARTIAL) are added in split order, x += that sum is written
// back, and the norm is taken of the updated row. Every load of a row is issued before the first
// add (the row's bytes are one round trip), which is what bounds this kernel. Rows are
// row0 + blockIdx.x.
constexpr int NORM_THREADS = 1024;
constexpr int NORM_VEC = 2;
constexpr int kMaxPartialSplits = 8;  // the host never splits K more than this

// L2-cached 16-byte load that yields zeros when `pred` is false. Volatile: a run of these is
// issued back to back, so all of them are in flight before the first use.
__device__ __forceinline__ float4 ldcg4_if(const float* p, bool pred) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  asm volatile(
      "{\n\t.reg .pred q;\n\tsetp.ne.b32 q, %5, 0;\n\t@q ld.global.cg.v4.f32 {%0,%1,%2,%3}, [%4];\n\t}"
      : "+f"(v.x), "+f"(v.y), "+f"(v.z), "+f"(v.w)
      : "l"(p), "r"((int)pred)
      : "memory");
  return v;
}

// Four L2-cached 16-byte loads p, p + stride, p + 2 stride, p + 3 stride (floats) in one asm
// statement: all four are issued before any of their results is used; load k is skipped (zeros)
// when k >= n.
__device__ __forceinline__ void ldcg4x4(const float* p, size_t stride, int n, float4 (&q)[4]) {
#pragma unroll
  for (int k = 0; k < 4; ++k) q[k] = make_float4(0.f, 0.f, 0.f, 0.f);
  asm volatile(
      "{\n\t.reg .pred p0, p1, p2, p3;\n\t"
      "setp.gt.s32 p0, %20, 0;\n\tsetp.gt.s32 p1, %20, 1;\n\tsetp.gt.s32 p2, %20, 2;\n\tsetp.gt.s32 p3, %20, 3;\n\t"
      "@p0 ld.global.cg.v4.f32 {%0,%1,%2,%3}, [%16];\n\t"
      "@p1 ld.global.cg.v4.f32 {%4,%5,%6,%7}, [%17];\n\t"
      "@p2 ld.global.cg.v4.f32 {%8,%9,%10,%11}, [%18];\n\t"
      "@p3 ld.global.cg.v4.f32 {%12,%13,%14,%15}, [%19];\n\t}"
      : "+f"(q[0].x), "+f"(q[0].y), "+f"(q[0].z), "+f"(q[0].w), "+f"(q[1].x), "+f"(q[1].y), "+f"(q[1].z), "+f"(q[1].w),
        "+f"(q[2].x), "+f"(q[2].y), "+f"(q[2].z), "+f"(q[2].w), "+f"(q[3].x), "+f"(q[3].y), "+f"(q[3].z), "+f"(q[3].w)
      : "l"(p), "l"(p + stride), "l"(p + 2 * stride), "l"(p + 3 * stride), "r"(n)
      : "memory");
}

__device__ __forceinline__ void store4(float* y, float4 v) { *reinterpret_cast<float4*>(y) = v; }
// four values rounded to bf16, then converted to fp16 (exact for magnitudes in [2^-14, 65504];
// smaller ones keep fp16's subnormal spacing 2^-24), stored as fp16 bit patterns
__device__ __forceinline__ void store4_bf16_as_f16(bf16* y, float4 v) {
  const __half2 lo = __floats2half2_rn(__bfloat162float(__float2bfloat16_rn(v.x)),
                                       __bfloat162float(__float2bfloat16_rn(v.y)));
  const __half2 hi = __floats2half2_rn(__bfloat162float(__float2bfloat16_rn(v.z)),
                                       __bfloat162float(__float2bfloat16_rn(v.w)));
  *reinterpret_cast<uint2*>(y) = make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                                            *reinterpret_cast<const uint32_t*>(&hi));
}
__device__ __forceinline__ void store4(bf16* y, float4 v) {
  const uint32_t lo = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v.x)) |
                      ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v.y)) << 16);
  const uint32_t hi = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v.z)) |
                      ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v.w)) << 16);
  *reinterpret_cast<uint2*>(y) = make_uint2(lo, hi);
}

template <typename T, int KS>
__global__ void __launch_bounds__(NORM_THREADS) k_rmsnorm(float* __restrict__ x, const float* __restrict__ gain,
                                                          T* __restrict__ y, int d, float eps, SplitPartials sp,
                                                          int row0) {
  __shared__ float red[NORM_THREADS / 32];
  JF_TL_ENTRY();
  pdl_launch_dependents();  // the next projection may launch now and prefetch its weights
  const int nv = d >> 2;
  // the gains are weights (written before this forward began): fetched before the dependency wait
  const float4* g4 = reinterpret_cast<const float4*>(gain);
  float4 gv[NORM_VEC];
#pragma unroll
  for (int j = 0; j < NORM_VEC; ++j) {
    const int i = threadIdx.x + j * NORM_THREADS;
    gv[j] = (i < nv) ? g4[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  pdl_wait();
  JF_TL_WAITED();
  const int r = row0 + blockIdx.x;
  float4* xr = reinterpret_cast<float4*>(x + (size_t)r * d);
  float4 v[NORM_VEC];
#pragma unroll
  for (int j = 0; j < NORM_VEC; ++j) {
    const int i = threadIdx.x + j * NORM_THREADS;
    v[j] = (i < nv) ? xr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  if constexpr (KS > 0) {
    // the KS split partials of a vector: KS independent loads, then added in split order
#pragma unroll
    for (int j = 0; j < NORM_VEC; ++j) {
      if (j * NORM_THREADS >= nv) break;
      const int i = threadIdx.x + j * NORM_THREADS;
      if (i < nv) {
        const int n = 4 * i;
        const float* base = sp.ws + ((size_t)((n >> 7) * sp.m_tiles + r / sp.bn) * KS * sp.bn +
                                     (size_t)(r % sp.bn)) * 128 + (n & 127);
        constexpr int NB = (KS + 3) / 4;
        float4 q[NB][4];
        const size_t stride = (size_t)sp.bn * 128;
#pragma unroll
        for (int b = 0; b < NB; ++b) ldcg4x4(base + (size_t)(4 * b) * stride, stride, KS - 4 * b, q[b]);
        float4 acc = q[0][0];
#pragma unroll
        for (int s = 1; s < KS; ++s) {
          acc.x += q[s >> 2][s & 3].x;
          acc.y += q[s >> 2][s & 3].y;
          acc.z += q[s >> 2][s & 3].z;
          acc.w += q[s >> 2][s & 3].w;
        }
        v[j] = make_float4(v[j].x + acc.x, v[j].y + acc.y, v[j].z + acc.z, v[j].w + acc.w);
        xr[i] = v[j];
      }
    }
  }
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < NORM_VEC; ++j) {
    ss = fmaf(v[j].x, v[j].x, ss);
    ss = fmaf(v[j].y, v[j].y, ss);
    ss = fmaf(v[j].z, v[j].z, ss);
    ss = fmaf(v[j].w, v[j].w, ss);
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < NORM_THREADS / 32; ++w) tot += red[w];
  const float rs = 1.0f / sqrtf(tot / (float)d + eps);
  T* yr = y + (size_t)blockIdx.x * d;
#pragma unroll
  for (int j = 0; j < NORM_VEC; ++j) {
    const int i = threadIdx.x + j * NORM_THREADS;
    if (i < nv) {
      const float4 g = gv[j];
      store4(yr + 4 * i, make_float4(v[j].x * rs * g.x, v[j].y * rs * g.y, v[j].z * rs * g.z, v[j].w * rs * g.w));
    }
  }
  JF_TL_EXIT(KS > 0 ? TL_NORM_ACC : TL_NORM);
}

// Finish of the QKV projection from its split-K partials (EPI_PARTIAL, head_dim 128 = one weight
// tile per head): for row m and head slot hs (query heads, then key heads, then value heads), add
// the partials in split order, then the feature's bias when the model has QKV biases, rotate query and key heads by the row's position (rotate-half RoPE,
// the same arithmetic as the fused epilogue), round to bf16 and store to q [m][Hq][128],
// k / v [m][Hkv][128] (v as fp16 values of the bf16-rounded numbers). One warp per (row, head slot); lane l holds dims 4l .. 4l+3, whose rotation
// partner is lane l ^ 16.
__global__ void __launch_bounds__(128) k_qkv_finish(SplitPartials sp, const bf16* __restrict__ bias,
                                                     const int* __restrict__ pos,
                                                     const float2* __restrict__ rope, bf16* __restrict__ q,
                                                     bf16* __restrict__ k, bf16* __restrict__ v, int M, int Hq,
                                                     int Hkv) {
  JF_TL_ENTRY();
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int slots = Hq + 2 * Hkv;
  const int job = blockIdx.x * 4 + warp;
  if (job >= M * slots) return;
  const int m = job / slots, hs = job % slots;
  const bool rot = hs < Hq + Hkv;
  // before the dependency wait: the bias (a weight), the row's position (written before this
  // forward's kernels: by a host copy, or by the state machine after the previous forward) and its
  // rotary coefficients (a table built at context creation)
  uint2 bw = make_uint2(0u, 0u);
  if (bias != nullptr) bw = *reinterpret_cast<const uint2*>(bias + (size_t)hs * 128 + lane * 4);
  float2 c0 = make_float2(1.f, 0.f), c1 = c0, c2 = c0, c3 = c0;
  if (rot) {
    const float2* cs = rope + (size_t)pos[m] * 64 + ((lane * 4) & 63);
    c0 = cs[0];
    c1 = cs[1];
    c2 = cs[2];
    c3 = cs[3];
  }
  pdl_wait();
  JF_TL_WAITED();
  const float* base = sp.ws + ((size_t)(hs * sp.m_tiles + m / sp.bn) * sp.k_splits * sp.bn + (size_t)(m % sp.bn)) * 128 +
                      lane * 4;
  // all partials in flight at once, then added in split order
  float4 t[kMaxPartialSplits];
#pragma unroll
  for (int s = 0; s < kMaxPartialSplits; ++s)
    t[s] = ldcg4_if(base + (size_t)s * sp.bn * 128, s < sp.k_splits);
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int s = 0; s < kMaxPartialSplits; ++s) {
    if (s < sp.k_splits) {
      a.x += t[s].x;
      a.y += t[s].y;
      a.z += t[s].z;
      a.w += t[s].w;
    }
  }
  if (bias != nullptr) {  // per-feature bias (bf16 values), after the projection, before RoPE
    a.x += __uint_as_float(bw.x << 16);
    a.y += __uint_as_float(bw.x & 0xffff0000u);
    a.z += __uint_as_float(bw.y << 16);
    a.w += __uint_as_float(bw.y & 0xffff0000u);
  }
  bf16* dst;
  if (rot) {
    const float4 b = make_float4(__shfl_xor_sync(0xffffffffu, a.x, 16), __shfl_xor_sync(0xffffffffu, a.y, 16),
                                 __shfl_xor_sync(0xffffffffu, a.z, 16), __shfl_xor_sync(0xffffffffu, a.w, 16));
    if (lane < 16) {
      a = make_float4(a.x * c0.x - b.x * c0.y, a.y * c1.x - b.y * c1.y, a.z * c2.x - b.z * c2.y, a.w * c3.x - b.w * c3.y);
    } else {
      a = make_float4(a.x * c0.x + b.x * c0.y, a.y * c1.x + b.y * c1.y, a.z * c2.x + b.z * c2.y, a.w * c3.x + b.w * c3.y);
    }
    dst = (hs < Hq) ? q + ((size_t)m * Hq + hs) * 128 : k + ((size_t)m * Hkv + (hs - Hq)) * 128;
    store4(dst + lane * 4, a);
  } else {
    // values: rounded to bf16 (the model's rounding point), then stored as fp16, the type the
    // attention's P V product reads them in (exact for magnitudes in fp16's normal range)
    dst = v + ((size_t)m * Hkv + (hs - Hq - Hkv)) * 128;
    store4_bf16_as_f16(dst + lane * 4, a);
  }
  JF_TL_EXIT(TL_QKV_FINISH);
}

template <typename K, typename... Args>
cudaError_t launch_pdl(K kernel, dim3 grid, dim3 block, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

}  // namespace

#ifdef JF_TIMELINE
JF_TL_SETTER(tl_set_elem)
#endif

// Wait-limit probe: one thread waits, under the given limit, on a shared-memory mbarrier that
// nothing arrives at (no copy and no MMA is in flight), then stores how long it waited, records
// JF_DERR_TIMEOUT_PROBE in the error word and exits. It exercises the same bounded wait and
// error path as the kernels' waits on copies and MMAs, without leaving any operation behind.
__global__ void k_wait_probe(int* err, unsigned long long* waited_ns, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_u32(&bar);
  mbar_init(b, 1);
  fence_mbar_init();
  const uint64_t t0 = jf_globaltimer();
  const bool arrived = mbar_wait_bounded(b, 0u, limit_ns);
  *waited_ns = jf_globaltimer() - t0;
  if (!arrived) jf_set_error(err, JF_DERR_TIMEOUT_PROBE);
}

cudaError_t launch_wait_probe(int* err, unsigned long long* waited_ns, unsigned long long limit_ns, cudaStream_t st) {
  k_wait_probe<<<1, 1, 0, st>>>(err, waited_ns, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_init_weights(void* dst, bool is_bf16, long long rows, long long cols, uint64_t seed, uint64_t tid,
                                double stdv, long long grp, long long grp_stride, long long grp_off, cudaStream_t st) {
  const long long npairs = (rows * cols + 1) / 2;
  long long blocks = (npairs + 255) / 256;
  if (blocks > 152 * 64) blocks = 152 * 64;
  if (blocks < 1) blocks = 1;
  if (is_bf16)
    k_init_weights<bf16><<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<bf16*>(dst), rows, cols, seed, tid, stdv,
                                                           grp, grp_stride, grp_off);
  else
    k_init_weights<float><<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<float*>(dst), rows, cols, seed, tid,
                                                            stdv, grp, grp_stride, grp_off);
  return cudaGetLastError();
}

cudaError_t launch_fill_f32(float* p, long long n, float v, cudaStream_t st) {
  long long blocks = (n + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  k_fill_f32<<<(unsigned)blocks, 256, 0, st>>>(p, n, v);
  return cudaGetLastError();
}

cudaError_t launch_rope_table(float2* tab, int n_pos, int half, double theta, cudaStream_t st) {
  long long n = (long long)n_pos * half;
  long long blocks = (n + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  k_rope_table<<<(unsigned)blocks, 256, 0, st>>>(tab, n_pos, half, theta);
  return cudaGetLastError();
}

cudaError_t launch_embed(const void* E, bool is_bf16, const int* tok, float* x, int rows, int d, int V, int* err,
                         cudaStream_t st) {
  if (is_bf16)
    return launch_pdl(k_embed<bf16>, dim3(rows), dim3(256), st, reinterpret_cast<const bf16*>(E), tok, x, d, V, err);
  return launch_pdl(k_embed<float>, dim3(rows), dim3(256), st, reinterpret_cast<const float*>(E), tok, x, d, V, err);
}

template <int KS>
cudaError_t launch_rmsnorm_ks(float* x, const float* gain, bf16* y, int rows, int d, float eps,
                              const SplitPartials& sp, int row0, cudaStream_t st) {
  return launch_pdl(k_rmsnorm<bf16, KS>, dim3(rows), dim3(NORM_THREADS), st, x, gain, y, d, eps, sp, row0);
}

cudaError_t launch_rmsnorm(float* x, const float* gain, void* y, bool is_bf16, int rows, int d, float eps,
                           const SplitPartials* acc, int row0, cudaStream_t st) {
  const SplitPartials sp = acc ? *acc : SplitPartials{nullptr, 0, 1, 1};
  if (is_bf16) {
    bf16* yb = reinterpret_cast<bf16*>(y);
    switch (acc ? sp.k_splits : 0) {
      case 0: return launch_rmsnorm_ks<0>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 1: return launch_rmsnorm_ks<1>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 2: return launch_rmsnorm_ks<2>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 3: return launch_rmsnorm_ks<3>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 4: return launch_rmsnorm_ks<4>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 5: return launch_rmsnorm_ks<5>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 6: return launch_rmsnorm_ks<6>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 7: return launch_rmsnorm_ks<7>(x, gain, yb, rows, d, eps, sp, row0, st);
      case 8: return launch_rmsnorm_ks<8>(x, gain, yb, rows, d, eps, sp, row0, st);
      default: return cudaErrorInvalidValue;
    }
  }
  if (acc) return cudaErrorInvalidValue;
  return launch_pdl(k_rmsnorm<float, 0>, dim3(rows), dim3(NORM_THREADS), st, x, gain, reinterpret_cast<float*>(y),
                    d, eps, sp, row0);
}

cudaError_t launch_qkv_finish(const SplitPartials& sp, const void* bias, const int* pos, const float2* rope, void* q,
                              void* k, void* v, int M, int Hq, int Hkv, cudaStream_t st) {
  const int jobs = M * (Hq + 2 * Hkv);
  return launch_pdl(k_qkv_finish, dim3((jobs + 3) / 4), dim3(128), st, sp, reinterpret_cast<const bf16*>(bias), pos,
                    rope, reinterpret_cast<bf16*>(q),
                    reinterpret_cast<bf16*>(k), reinterpret_cast<bf16*>(v), M, Hq, Hkv);
}

}  // namespace jf
