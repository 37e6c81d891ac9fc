// Attention of the in-flight rows over the exact committed KV cache (Sec. 2.1, Eq. 3: the
// block's n conditionals come out of one pass with a causal mask) and the block-causal tree mask
// of multi-block decoding and rejection recycling (Sec. 3.2, Algorithm 1).
//
// Rows are grouped into chains (jf_internal.h): a chain's rows sit at consecutive positions
// starting at the sequence's committed length P, and a row at position p attends to cache
// positions [0, P) and to the chain's own rows at positions P .. p. A real-active draft followed
// by its pseudo-active blocks is one chain; each recycled candidate is a chain of its own. Hence
// every row attends to exactly the positions 0 .. p, each position resolved either to a KV page
// (p < P) or to an in-flight row of its chain.
//
// bf16 path: split-KV flash decoding. Work unit = (chain, KV head, tile of 64 (token, head)
// query rows); items = (unit, chunk of 128 key positions aligned at multiples of 128). Each item
// runs QK^T and PV on mma.sync.m16n8k16 with an online softmax, keys staged by cp.async into
// XOR-swizzled shared memory. Partials are merged in chunk order by the unit's last item
// (atomic ticket). Chunk boundaries are absolute, so a row's arithmetic depends only on its own
// key set and not on how many rows share the forward.
// fp32 path: one warp per (row, head), keys in absolute order, online softmax in fp32.
#include "jf_device.cuh"
#include "jf_internal.h"

namespace jf {
namespace {

constexpr int HD = 128;
constexpr int SUB = 64;                   // keys per sub-block
constexpr int NSUB = kAttnChunk / SUB;    // sub-blocks per chunk
constexpr int ROW_BYTES = HD * 2;         // 256 bytes per key / query row
constexpr int TILE_BYTES = SUB * ROW_BYTES;  // 16 KB

JF_DEV uint32_t swz(int r, int c16) { return (uint32_t)(r * ROW_BYTES + ((c16 ^ (r & 7)) << 4)); }

JF_DEV void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}
JF_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
JF_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

JF_DEV void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
JF_DEV void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

JF_DEV void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

JF_DEV uint32_t pack_bf16(float lo, float hi) {
  const bf16 l = __float2bfloat16_rn(lo), h = __float2bfloat16_rn(hi);
  return (uint32_t)__bfloat16_as_ushort(l) | ((uint32_t)__bfloat16_as_ushort(h) << 16);
}

// Address of the K (or V) row for absolute key position kp of unit (chain, kvh); null if the
// position holds no key for this chain. spage: the chunk's page ids (kp0 / 16 ...), resolved once.
JF_DEV const bf16* key_row(const AttnParams& a, const bf16* pages, const bf16* inf, const Chain& ch, int kvh, int kp,
                           int max_kp, int kp0, const int* spage) {
  if (kp > max_kp) return nullptr;
  if (kp < ch.pos0) {
    const int page = spage[(kp - kp0) >> 4];
    if (page < 0 || page >= a.n_pages) return nullptr;
    return pages + (((size_t)page * a.Hkv + kvh) * kPage + (kp & 15)) * HD;
  }
  return inf + ((size_t)(ch.row0 + kp - ch.pos0) * a.Hkv + kvh) * HD;
}

// One work item = (unit, 128-key chunk). 8 warps: warp w computes query-row group w & 3 (16 rows)
// against key sub-block w >> 2 (64 keys); the two sub-block partials of a row are merged in shared
// memory, sub-block 0 first, so the chunk's arithmetic is fixed by absolute key positions.
constexpr int ATT_THREADS = 256;

__global__ void __launch_bounds__(ATT_THREADS, 1) k_attn_bf16(const AttnParams a) {
  extern __shared__ __align__(128) uint8_t sm[];
  uint8_t* sQ = sm;                       // 64 x 256 B
  uint8_t* sK = sm + TILE_BYTES;          // NSUB x 16 KB
  uint8_t* sV = sK + NSUB * TILE_BYTES;   // NSUB x 16 KB
  float* sO1 = reinterpret_cast<float*>(sK + TILE_BYTES);  // sub-block 1 partial O [64][128], reuses K1/V1
  __shared__ int s_rowpos[kAttnQRows];
  __shared__ int s_page[kAttnChunk / kPage];
  __shared__ float s_m1[kAttnQRows], s_l1[kAttnQRows];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rg = warp & 3, sb = warp >> 2;
  pdl_launch_dependents();  // the next kernel may launch now
  pdl_wait();
  const int n_items = a.plan->n_items;
  const int G = a.Hq / a.Hkv;
  const bf16* Kp = reinterpret_cast<const bf16*>(a.k_pages);
  const bf16* Vp = reinterpret_cast<const bf16*>(a.v_pages);
  const bf16* Ki = reinterpret_cast<const bf16*>(a.k_inf);
  const bf16* Vi = reinterpret_cast<const bf16*>(a.v_inf);
  const bf16* Q = reinterpret_cast<const bf16*>(a.q);
  bf16* Out = reinterpret_cast<bf16*>(a.out);

  for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
    const int2 it = a.items[item];
    const AttnUnit u = a.units[it.x];
    const int chunk = it.y;
    const Chain ch = a.chains[u.chain];
    const int nq = ch.nrows * G;
    const int qr0 = u.qt * kAttnQRows;
    int qrows = nq - qr0;
    if (qrows > kAttnQRows) qrows = kAttnQRows;
    const int max_kp = ch.pos0 + (qr0 + qrows - 1) / G;
    const int kp0 = chunk * kAttnChunk;

    if (tid < kAttnQRows) s_rowpos[tid] = (tid < qrows) ? ch.pos0 + (qr0 + tid) / G : -1;
    if (tid < kAttnChunk / kPage) {
      const int kp = kp0 + tid * kPage;
      s_page[tid] = (kp < ch.pos0) ? a.page_table[(size_t)ch.seq * a.pages_per_seq + (kp >> 4)] : -1;
    }
    // stage Q (64 rows, zero beyond qrows)
    for (int i = tid; i < kAttnQRows * 16; i += ATT_THREADS) {
      const int r = i >> 4, c = i & 15;
      const bool ok = r < qrows;
      const int qr = qr0 + (ok ? r : 0);
      const int t = qr / G, g = qr % G;
      const bf16* src = Q + ((size_t)(ch.row0 + t) * a.Hq + u.kvh * G + g) * HD + c * 8;
      cp_async16(smem_u32(sQ) + swz(r, c), src, ok);
    }
    __syncthreads();  // page ids visible
    // stage the chunk's keys and values
    for (int i = tid; i < NSUB * SUB * 16; i += ATT_THREADS) {
      const int r = i >> 4, c = i & 15;      // r: key within the chunk
      const int kp = kp0 + r;
      const bf16* kr = key_row(a, Kp, Ki, ch, u.kvh, kp, max_kp, kp0, s_page);
      const bf16* vr = key_row(a, Vp, Vi, ch, u.kvh, kp, max_kp, kp0, s_page);
      const int b = r / SUB, rr = r % SUB;
      cp_async16(smem_u32(sK + b * TILE_BYTES) + swz(rr, c), kr ? kr + c * 8 : Kp, kr != nullptr);
      cp_async16(smem_u32(sV + b * TILE_BYTES) + swz(rr, c), vr ? vr + c * 8 : Vp, vr != nullptr);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();

    // Q fragments of this warp's 16 rows
    uint32_t qf[HD / 16][4];
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const int r = rg * 16 + (lane & 15), c = kk * 2 + (lane >> 4);
      ldsm_x4(smem_u32(sQ) + swz(r, c), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
    }
    const int r_lo = rg * 16 + (lane >> 2), r_hi = r_lo + 8;
    const int pos_lo = s_rowpos[r_lo], pos_hi = s_rowpos[r_hi];
    float o[HD / 8][4];
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

    const uint32_t kb = smem_u32(sK + sb * TILE_BYTES), vb = smem_u32(sV + sb * TILE_BYTES);
    float s[SUB / 8][4];
#pragma unroll
    for (int nt = 0; nt < SUB / 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < SUB / 16; ++np) {
        uint32_t b0, b1, b2, b3;
        const int r = np * 16 + (lane & 7) + ((lane >> 4) << 3), c = kk * 2 + ((lane >> 3) & 1);
        ldsm_x4(kb + swz(r, c), b0, b1, b2, b3);
        mma16816(s[2 * np], qf[kk], b0, b1);
        mma16816(s[2 * np + 1], qf[kk], b2, b3);
      }
    }
    // mask (key position <= row position); softmax statistics of this 64-key sub-block (log2 domain)
    const int kbase = kp0 + sb * SUB + 2 * (lane & 3);
    float m_lo = -INFINITY, m_hi = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < SUB / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int kp = kbase + nt * 8 + e;
        s[nt][e] = (kp <= pos_lo) ? s[nt][e] * a.scale_log2 : -INFINITY;
        s[nt][2 + e] = (kp <= pos_hi) ? s[nt][2 + e] * a.scale_log2 : -INFINITY;
        m_lo = fmaxf(m_lo, s[nt][e]);
        m_hi = fmaxf(m_hi, s[nt][2 + e]);
      }
    }
#pragma unroll
    for (int sh = 1; sh <= 2; sh <<= 1) {
      m_lo = fmaxf(m_lo, __shfl_xor_sync(0xffffffffu, m_lo, sh));
      m_hi = fmaxf(m_hi, __shfl_xor_sync(0xffffffffu, m_hi, sh));
    }
    const float b_lo = (m_lo == -INFINITY) ? 0.f : m_lo;
    const float b_hi = (m_hi == -INFINITY) ? 0.f : m_hi;
    float l_lo = 0.f, l_hi = 0.f;
#pragma unroll
    for (int nt = 0; nt < SUB / 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - b_lo);
      s[nt][1] = exp2f(s[nt][1] - b_lo);
      s[nt][2] = exp2f(s[nt][2] - b_hi);
      s[nt][3] = exp2f(s[nt][3] - b_hi);
      l_lo += s[nt][0] + s[nt][1];
      l_hi += s[nt][2] + s[nt][3];
    }
    // O = P V
#pragma unroll
    for (int kj = 0; kj < SUB / 16; ++kj) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kj][0], s[2 * kj][1]);
      pa[1] = pack_bf16(s[2 * kj][2], s[2 * kj][3]);
      pa[2] = pack_bf16(s[2 * kj + 1][0], s[2 * kj + 1][1]);
      pa[3] = pack_bf16(s[2 * kj + 1][2], s[2 * kj + 1][3]);
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        uint32_t b0, b1, b2, b3;
        const int r = kj * 16 + (lane & 7) + (((lane >> 3) & 1) << 3), c = dp * 2 + (lane >> 4);
        ldsm_x4_t(vb + swz(r, c), b0, b1, b2, b3);
        mma16816(o[2 * dp], pa, b0, b1);
        mma16816(o[2 * dp + 1], pa, b2, b3);
      }
    }
#pragma unroll
    for (int sh = 1; sh <= 2; sh <<= 1) {
      l_lo += __shfl_xor_sync(0xffffffffu, l_lo, sh);
      l_hi += __shfl_xor_sync(0xffffffffu, l_hi, sh);
    }
    const int d0 = 2 * (lane & 3);
    __syncthreads();  // every warp is done with K/V: sub-block 1 partials may overwrite them
    if (sb == 1) {
#pragma unroll
      for (int i = 0; i < HD / 8; ++i) {
        *reinterpret_cast<float2*>(sO1 + r_lo * HD + i * 8 + d0) = make_float2(o[i][0], o[i][1]);
        *reinterpret_cast<float2*>(sO1 + r_hi * HD + i * 8 + d0) = make_float2(o[i][2], o[i][3]);
      }
      if ((lane & 3) == 0) {
        s_m1[r_lo] = m_lo;
        s_l1[r_lo] = l_lo;
        s_m1[r_hi] = m_hi;
        s_l1[r_hi] = l_hi;
      }
    }
    __syncthreads();
    if (sb == 0) {
      // merge: m = max(m0, m1), O = 2^(m0-m) O0 + 2^(m1-m) O1, l likewise
      const float m1_lo = s_m1[r_lo], m1_hi = s_m1[r_hi];
      const float mm_lo = fmaxf(m_lo, m1_lo), mm_hi = fmaxf(m_hi, m1_hi);
      const float a0_lo = (m_lo == -INFINITY) ? 0.f : exp2f(m_lo - mm_lo);
      const float a1_lo = (m1_lo == -INFINITY) ? 0.f : exp2f(m1_lo - mm_lo);
      const float a0_hi = (m_hi == -INFINITY) ? 0.f : exp2f(m_hi - mm_hi);
      const float a1_hi = (m1_hi == -INFINITY) ? 0.f : exp2f(m1_hi - mm_hi);
      l_lo = a0_lo * l_lo + a1_lo * s_l1[r_lo];
      l_hi = a0_hi * l_hi + a1_hi * s_l1[r_hi];
#pragma unroll
      for (int i = 0; i < HD / 8; ++i) {
        const float2 p_lo = *reinterpret_cast<const float2*>(sO1 + r_lo * HD + i * 8 + d0);
        const float2 p_hi = *reinterpret_cast<const float2*>(sO1 + r_hi * HD + i * 8 + d0);
        o[i][0] = a0_lo * o[i][0] + a1_lo * p_lo.x;
        o[i][1] = a0_lo * o[i][1] + a1_lo * p_lo.y;
        o[i][2] = a0_hi * o[i][2] + a1_hi * p_hi.x;
        o[i][3] = a0_hi * o[i][3] + a1_hi * p_hi.y;
      }
      m_lo = mm_lo;
      m_hi = mm_hi;
      if (u.n_chunks == 1) {
        const float il_lo = l_lo > 0.f ? 1.f / l_lo : 0.f, il_hi = l_hi > 0.f ? 1.f / l_hi : 0.f;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int r = half ? r_hi : r_lo;
          if (r >= qrows) continue;
          const float il = half ? il_hi : il_lo;
          const int qr = qr0 + r, t = qr / G, g = qr % G;
          bf16* dst = Out + ((size_t)(ch.row0 + t) * a.Hq + u.kvh * G + g) * HD;
#pragma unroll
          for (int i = 0; i < HD / 8; ++i) {
            const float x0 = o[i][2 * half] * il, x1 = o[i][2 * half + 1] * il;
            *reinterpret_cast<uint32_t*>(dst + i * 8 + d0) = pack_bf16(x0, x1);
          }
        }
      } else {
        const int slot = u.slot0 + chunk;
        float* wo = a.ws_o + (size_t)slot * kAttnQRows * HD;
        float* wml = a.ws_ml + (size_t)slot * kAttnQRows * 2;
#pragma unroll
        for (int i = 0; i < HD / 8; ++i) {
          *reinterpret_cast<float2*>(wo + r_lo * HD + i * 8 + d0) = make_float2(o[i][0], o[i][1]);
          *reinterpret_cast<float2*>(wo + r_hi * HD + i * 8 + d0) = make_float2(o[i][2], o[i][3]);
        }
        if ((lane & 3) == 0) {
          wml[r_lo * 2] = m_lo;
          wml[r_lo * 2 + 1] = l_lo;
          wml[r_hi * 2] = m_hi;
          wml[r_hi * 2 + 1] = l_hi;
        }
      }
    }
    __syncthreads();
  }
}

// Merge of the split-KV partials of multi-chunk units, in chunk order:
//   out = sum_c 2^(m_c - M) O_c / sum_c 2^(m_c - M) l_c,  M = max_c m_c.
// CTA (x, u) handles rows 8x .. 8x+7 of unit u; thread = (row, 4 of the 128 dims).
__global__ void __launch_bounds__(256) k_attn_combine(const AttnParams a) {
  pdl_launch_dependents();
  pdl_wait();
  const int u_idx = blockIdx.y;
  if (u_idx >= a.plan->n_units) return;
  const AttnUnit u = a.units[u_idx];
  if (u.n_chunks == 1) return;
  const Chain ch = a.chains[u.chain];
  const int G = a.Hq / a.Hkv;
  const int qr0 = u.qt * kAttnQRows;
  int qrows = ch.nrows * G - qr0;
  if (qrows > kAttnQRows) qrows = kAttnQRows;
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (r >= qrows) return;
  const int d = (threadIdx.x & 31) * 4;
  const float2* ml = reinterpret_cast<const float2*>(a.ws_ml);
  float M = -INFINITY;
#pragma unroll 4
  for (int c = 0; c < u.n_chunks; ++c) M = fmaxf(M, __ldcg(ml + (size_t)(u.slot0 + c) * kAttnQRows + r).x);
  float L = 0.f, acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
#pragma unroll 4
  for (int c = 0; c < u.n_chunks; ++c) {
    const size_t sl = (size_t)(u.slot0 + c);
    const float2 p = __ldcg(ml + sl * kAttnQRows + r);
    const float4 oc = __ldcg(reinterpret_cast<const float4*>(a.ws_o + (sl * kAttnQRows + r) * HD + d));
    const float w = (p.x == -INFINITY) ? 0.f : exp2f(p.x - M);
    L += w * p.y;
    acc0 += w * oc.x;
    acc1 += w * oc.y;
    acc2 += w * oc.z;
    acc3 += w * oc.w;
  }
  const float il = L > 0.f ? 1.f / L : 0.f;
  const int qr = qr0 + r, t = qr / G, g = qr % G;
  bf16* dst = reinterpret_cast<bf16*>(a.out) + ((size_t)(ch.row0 + t) * a.Hq + u.kvh * G + g) * HD + d;
  *reinterpret_cast<uint32_t*>(dst) = pack_bf16(acc0 * il, acc1 * il);
  *reinterpret_cast<uint32_t*>(dst + 2) = pack_bf16(acc2 * il, acc3 * il);
}

// fp32 path: one warp per (row, query head); keys in absolute order, 32 at a time.
__global__ void __launch_bounds__(128) k_attn_f32(const AttnParams a, int n_rows) {
  const int warp_global = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  pdl_wait();
  const int r = warp_global / a.Hq, h = warp_global % a.Hq;
  if (r >= n_rows) return;
  const int hd = a.hd, G = a.Hq / a.Hkv, kvh = h / G;
  const int n_ch = *a.n_chains_dev;
  int ci = 0;
  for (; ci < n_ch; ++ci) {
    const Chain c = a.chains[ci];
    if (r >= c.row0 && r < c.row0 + c.nrows) break;
  }
  if (ci == n_ch) return;
  const Chain ch = a.chains[ci];
  const int pos = ch.pos0 + (r - ch.row0);
  const float* q = reinterpret_cast<const float*>(a.q) + ((size_t)r * a.Hq + h) * hd;
  const float* Kp = reinterpret_cast<const float*>(a.k_pages);
  const float* Vp = reinterpret_cast<const float*>(a.v_pages);
  const float* Ki = reinterpret_cast<const float*>(a.k_inf);
  const float* Vi = reinterpret_cast<const float*>(a.v_inf);
  const float scale = a.scale_log2;
  float m = -INFINITY, l = 0.f, o0 = 0.f, o1 = 0.f;
  for (int kb = 0; kb <= pos; kb += 32) {
    const int kp = kb + lane;
    float s = -INFINITY;
    const float* kr = nullptr;
    const float* vr = nullptr;
    if (kp <= pos) {
      if (kp < ch.pos0) {
        const int page = a.page_table[(size_t)ch.seq * a.pages_per_seq + (kp >> 4)];
        const size_t off = (((size_t)page * a.Hkv + kvh) * kPage + (kp & 15)) * hd;
        kr = Kp + off;
        vr = Vp + off;
      } else {
        const size_t off = ((size_t)(ch.row0 + kp - ch.pos0) * a.Hkv + kvh) * hd;
        kr = Ki + off;
        vr = Vi + off;
      }
      float dot = 0.f;
      for (int i = 0; i < hd; ++i) dot = fmaf(q[i], kr[i], dot);
      s = dot * scale;
    }
    float mx = s;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    const float mn = fmaxf(m, mx);
    const float al = (m == -INFINITY) ? 0.f : exp2f(m - mn);
    const float p = (s == -INFINITY) ? 0.f : exp2f(s - mn);
    float ps = warp_sum(p);
    l = l * al + ps;
    o0 *= al;
    o1 *= al;
    for (int j = 0; j < 32; ++j) {
      const float pj = __shfl_sync(0xffffffffu, p, j);
      const int kpj = kb + j;
      if (kpj > pos) break;
      const float* vrow;
      if (kpj < ch.pos0) {
        const int page = a.page_table[(size_t)ch.seq * a.pages_per_seq + (kpj >> 4)];
        vrow = Vp + (((size_t)page * a.Hkv + kvh) * kPage + (kpj & 15)) * hd;
      } else {
        vrow = Vi + ((size_t)(ch.row0 + kpj - ch.pos0) * a.Hkv + kvh) * hd;
      }
      o0 = fmaf(pj, vrow[lane], o0);
      if (lane + 32 < hd) o1 = fmaf(pj, vrow[lane + 32], o1);
    }
    m = mn;
    (void)vr;
  }
  float* out = reinterpret_cast<float*>(a.out) + ((size_t)r * a.Hq + h) * hd;
  const float il = l > 0.f ? 1.f / l : 0.f;
  out[lane] = o0 * il;
  if (lane + 32 < hd) out[lane + 32] = o1 * il;
}

// Work decomposition of the bf16 attention for the current chains (one CTA, once per forward).
__global__ void k_attn_plan(const Chain* chains, const int* n_chains_dev, int Hq, int Hkv, AttnPlan* plan,
                            AttnUnit* units, int2* items, int max_units, int max_items, int max_slots, int* err) {
  pdl_launch_dependents();
  pdl_wait();
  if (threadIdx.x != 0) return;
  const int G = Hq / Hkv;
  int nu = 0, ni = 0, ns = 0;
  const int n_ch = *n_chains_dev;
  for (int c = 0; c < n_ch; ++c) {
    const Chain ch = chains[c];
    const int nq = ch.nrows * G;
    const int nqt = (nq + kAttnQRows - 1) / kAttnQRows;
    for (int kvh = 0; kvh < Hkv; ++kvh)
      for (int qt = 0; qt < nqt; ++qt) {
        int qrows = nq - qt * kAttnQRows;
        if (qrows > kAttnQRows) qrows = kAttnQRows;
        const int max_kp = ch.pos0 + (qt * kAttnQRows + qrows - 1) / G;
        const int nch = max_kp / kAttnChunk + 1;
        if (nu >= max_units || ni + nch > max_items || (nch > 1 && ns + nch > max_slots)) {
          jf_set_error(err, JF_DERR_BOUNDS);
          plan->n_units = plan->n_items = 0;
          return;
        }
        units[nu] = AttnUnit{c, kvh, qt, nch, ns};
        for (int k = 0; k < nch; ++k) items[ni + k] = make_int2(nu, k);
        ni += nch;
        if (nch > 1) ns += nch;
        ++nu;
      }
  }
  plan->n_units = nu;
  plan->n_items = ni;
  plan->n_slots = ns;
}

}  // namespace

size_t attn_bf16_smem_bytes() { return (size_t)TILE_BYTES * (1 + 2 * NSUB); }

cudaError_t launch_attn_plan(const Chain* chains, const int* n_chains_dev, int Hq, int Hkv, AttnPlan* plan,
                             AttnUnit* units, int2* items, int max_units, int max_items, int max_slots, int* err,
                             cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1);
  cfg.blockDim = dim3(32);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_attn_plan, chains, n_chains_dev, Hq, Hkv, plan, units, items, max_units,
                            max_items, max_slots, err);
}

cudaError_t attn_prepare() {
  return cudaFuncSetAttribute(k_attn_bf16, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)attn_bf16_smem_bytes());
}

cudaError_t launch_attn_bf16(const AttnParams& a, int grid, cudaStream_t st) {
  const size_t smem = attn_bf16_smem_bytes();
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_attn_bf16, a);
}

cudaError_t launch_attn_combine(const AttnParams& a, int max_units, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kAttnQRows / 8, max_units);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_attn_combine, a);
}

cudaError_t launch_attn_f32(const AttnParams& a, int n_rows, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((n_rows * a.Hq + 3) / 4);
  cfg.blockDim = dim3(128);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_attn_f32, a, n_rows);
}

}  // namespace jf
