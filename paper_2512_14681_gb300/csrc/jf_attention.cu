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
// bf16 path: split-KV flash decoding with a fixed reduction tree. Work unit = (chain, KV head,
// tile of 128 (token, head) query rows). Key positions are cut into absolute 128-key chunks, and
// chunk c belongs to lane c mod 8. A unit runs on one 8-CTA cluster: CTA j walks the chunks of
// lane j in increasing order, 64 keys at a time, with one online-softmax state per row (QK^T and
// PV on mma.sync.m16n8k16, keys staged by cp.async into XOR-swizzled shared memory, the next chunk
// in flight while the current one computes). Each warp then stages its 16 rows' lane state as one
// block and sends it with a bulk copy into the shared memory of the CTA that owns those rows;
// once its 8 blocks have arrived (mbarrier transaction count) each CTA folds its rows' 8 lane
// states in lane order. The tree depends only on absolute key positions, never on
// how many rows share the forward or how many chunks a unit has, so a row's result is the same in
// every batch.
// fp32 path: one warp per (row, head), keys in absolute order, online softmax in fp32.
#include "jf_device.cuh"
#include "jf_internal.h"

namespace jf {
namespace {

constexpr int HD = 128;
constexpr int SUB = 64;                      // keys per sub-block (one online-softmax step)
constexpr int NSUB = kAttnChunk / SUB;       // sub-blocks per chunk
constexpr int ROW_BYTES = HD * 2;            // 256 bytes per key / query row
constexpr int TILE_BYTES = SUB * ROW_BYTES;  // 16 KB
constexpr int STAGE_BYTES = 2 * NSUB * TILE_BYTES;     // K and V of one chunk: 64 KB
constexpr int ROWS_PER_CTA = kAttnQRows / kAttnLanes;  // rows each CTA of a cluster folds (16)
constexpr int Q_BYTES = kAttnQRows * ROW_BYTES;         // staged queries: 32 KB
// lane-state block of 16 rows: O [16][128], then m [16], then l [16] (fp32)
constexpr int BLOCK_FLOATS = ROWS_PER_CTA * HD + 2 * ROWS_PER_CTA;
constexpr int BLOCK_BYTES = BLOCK_FLOATS * 4;          // 8320 B
constexpr int RECV_BYTES = kAttnLanes * BLOCK_BYTES;   // the 8 lanes' blocks of this CTA's rows
constexpr int REGION0 = RECV_BYTES > Q_BYTES ? RECV_BYTES : Q_BYTES;  // queries, later the lane states
constexpr int ATT_SMEM = REGION0 + 2 * STAGE_BYTES;   // 193 KB
static_assert(BLOCK_BYTES % 16 == 0 && kAttnLanes * BLOCK_BYTES <= 2 * STAGE_BYTES, "lane-state blocks");

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

// Fold of two softmax states (m, l, O) in the log2 domain: m = max(ma, mb),
// O = 2^(ma-m) Oa + 2^(mb-m) Ob, l likewise; an empty state has m = -inf and weight 0.
JF_DEV void fold_weights(float ma, float mb, float& wa, float& wb, float& m) {
  m = fmaxf(ma, mb);
  wa = (ma == -INFINITY) ? 0.f : exp2f(ma - m);
  wb = (mb == -INFINITY) ? 0.f : exp2f(mb - m);
}

JF_DEV void issue_kv(const AttnParams& a, const AttnUnit& u, int chunk, int li, int max_kp, const int* s_page,
                     uint8_t* stage, int part) {
  const bf16* Kp = reinterpret_cast<const bf16*>(a.k_pages);
  const bf16* Vp = reinterpret_cast<const bf16*>(a.v_pages);
  const bf16* Ki = reinterpret_cast<const bf16*>(a.k_inf);
  const bf16* Vi = reinterpret_cast<const bf16*>(a.v_inf);
  uint8_t* sK = stage;
  uint8_t* sV = stage + NSUB * TILE_BYTES;
  const int kp0 = chunk * kAttnChunk;
  for (int i = threadIdx.x; i < kAttnChunk * 16; i += blockDim.x) {
    const int r = i >> 4, c = i & 15;
    const int kp = kp0 + r;
    const bool cached = kp < u.pos0;
    if (!(part & (cached ? 1 : 2))) continue;
    const bf16* kr = nullptr;
    const bf16* vr = nullptr;
    if (kp <= max_kp) {
      if (cached) {
        const int page = s_page[li * (kAttnChunk / kPage) + (r >> 4)];
        if (page >= 0 && page < a.n_pages) {
          const size_t off = (((size_t)page * a.Hkv + u.kvh) * kPage + (kp & 15)) * HD;
          kr = Kp + off;
          vr = Vp + off;
        }
      } else {
        const size_t off = ((size_t)(u.row0 + kp - u.pos0) * a.Hkv + u.kvh) * HD;
        kr = Ki + off;
        vr = Vi + off;
      }
    }
    const int b = r / SUB, rr = r % SUB;
    cp_async16(smem_u32(sK + b * TILE_BYTES) + swz(rr, c), kr ? kr + c * 8 : Kp, kr != nullptr);
    cp_async16(smem_u32(sV + b * TILE_BYTES) + swz(rr, c), vr ? vr + c * 8 : Vp, vr != nullptr);
  }
}

constexpr int ATT_THREADS = 256;

// 8 warps: warp w owns query rows 16w .. 16w+15 of the tile and walks the lane's chunks, 64 keys
// at a time, with one online-softmax state; at the end it stores that lane state of its 16 rows
// into CTA w of the cluster, which folds rows 16w .. 16w+15 over the 8 lanes.
// At most 200 registers a thread (51,200 of the SM's 65,536): the CTAs of the QKV finish kernel
// still resident on an SM leave room for this one, so the clusters are placed while it runs.
__global__ void __maxnreg__(200) k_attn_bf16(const AttnParams a) {
  extern __shared__ __align__(128) uint8_t sm[];
  uint8_t* sQ = sm;                                  // 128 x 256 B, free once the queries are in registers
  float* recv = reinterpret_cast<float*>(sm);        // [8 lanes][block], aliases sQ
  uint8_t* stage0 = sm + REGION0;                    // chunk stages, 64 KB each; outgoing blocks at the end
  __shared__ __align__(8) uint64_t recv_bar;
  __shared__ int s_rowpos[kAttnQRows];
  __shared__ int s_page[kAttnLaneChunks * (kAttnChunk / kPage)];
  __shared__ AttnUnit s_unit;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int j = (int)cluster_rank();
  const int ui = (int)cluster_id_x();
  const int G = a.Hq / a.Hkv;
  pdl_launch_dependents();  // the next kernel may launch now
  if (tid == 0) {
    // receives the 8 lane-state blocks of this CTA's rows (one bulk copy from each CTA)
    mbar_init(smem_u32(&recv_bar), 1);
    fence_mbar_init();
  }
  // Before the dependency wait: the chain table, the page table and the cached keys were written
  // by host copies or by an earlier graph launch, all complete before this forward began.
  // Unit ui of the forward: chains in order, then KV heads, then 128-row query tiles.
  if (tid == 0) s_unit.pad = 0;
  __syncthreads();
  if (warp == 0) {
    const int n_ch = *a.n_chains_dev;
    int base = 0;
    for (int c0 = 0; c0 < n_ch; c0 += 32) {
      const int c = c0 + lane;
      Chain ch = {0, 0, 0, 0};
      int nqt = 0;
      if (c < n_ch) {
        ch = a.chains[c];
        nqt = (ch.nrows * G + kAttnQRows - 1) / kAttnQRows;
      }
      const int nu = a.Hkv * nqt;
      int incl = nu;
#pragma unroll
      for (int sh = 1; sh < 32; sh <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, sh);
        if (lane >= sh) incl += v;
      }
      const int first = base + incl - nu;
      if (nu > 0 && ui >= first && ui < base + incl) {
        const int k = ui - first, kvh = k / nqt, qt = k % nqt;
        int qrows = ch.nrows * G - qt * kAttnQRows;
        if (qrows > kAttnQRows) qrows = kAttnQRows;
        const int nch = (ch.pos0 + (qt * kAttnQRows + qrows - 1) / G) / kAttnChunk + 1;
        if (nch > kAttnLanes * kAttnLaneChunks) {
          if (j == 0) jf_set_error(a.err, JF_DERR_BOUNDS);
        } else {
          s_unit = AttnUnit{ch.seq, ch.row0, ch.nrows, ch.pos0, kvh, qt, nch, 1};
        }
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    // the launch must cover every unit
    if (lane == 0 && j == 0 && ui == (int)(gridDim.x / kAttnLanes) - 1 && base > ui + 1)
      jf_set_error(a.err, JF_DERR_BOUNDS);
  }
  __syncthreads();
  const AttnUnit u = s_unit;
  if (!u.pad) return;  // past the last unit: the whole cluster leaves together
  const int qr0 = u.qt * kAttnQRows;
  int qrows = u.nrows * G - qr0;
  if (qrows > kAttnQRows) qrows = kAttnQRows;
  const int max_kp = u.pos0 + (qr0 + qrows - 1) / G;
  const int n_lane = (u.n_chunks > j) ? (u.n_chunks - 1 - j) / kAttnLanes + 1 : 0;
  const int n_steps = n_lane;
  auto sub_of = [&](int t) { return j + kAttnLanes * t; };

  for (int i = tid; i < kAttnQRows; i += ATT_THREADS) s_rowpos[i] = (i < qrows) ? u.pos0 + (qr0 + i) / G : -1;
  for (int i = tid; i < n_lane * (kAttnChunk / kPage); i += ATT_THREADS) {
    const int li = i / (kAttnChunk / kPage), pg = i % (kAttnChunk / kPage);
    const int kp = (j + li * kAttnLanes) * kAttnChunk + pg * kPage;
    s_page[i] = (kp < u.pos0) ? a.page_table[(size_t)u.seq * a.pages_per_seq + (kp >> 4)] : -1;
  }
  __syncthreads();
  if (n_steps > 0) {
    issue_kv(a, u, sub_of(0), 0, max_kp, s_page, stage0, 1);
    cp_async_commit();
  }
  pdl_wait();  // queries and in-flight keys come from the QKV projection
  const bf16* Q = reinterpret_cast<const bf16*>(a.q);
  if (n_steps > 0) {
    for (int i = tid; i < kAttnQRows * 16; i += ATT_THREADS) {
      const int r = i >> 4, c = i & 15;
      const bool ok = r < qrows;
      const int qr = qr0 + (ok ? r : 0);
      const int t = qr / G, g = qr % G;
      const bf16* src = Q + ((size_t)(u.row0 + t) * a.Hq + u.kvh * G + g) * HD + c * 8;
      cp_async16(smem_u32(sQ) + swz(r, c), src, ok);
    }
    issue_kv(a, u, sub_of(0), 0, max_kp, s_page, stage0, 2);
    cp_async_commit();
    if (n_steps > 1) {
      issue_kv(a, u, sub_of(1), 1, max_kp, s_page, stage0 + STAGE_BYTES, 3);
      cp_async_commit();
    }
  }

  const int r_lo = warp * 16 + (lane >> 2), r_hi = r_lo + 8;
  const int pos_lo = s_rowpos[r_lo], pos_hi = s_rowpos[r_hi];
  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_lo = -INFINITY, m_hi = -INFINITY, l_lo = 0.f, l_hi = 0.f;
  uint32_t qf[HD / 16][4];

  for (int t = 0; t < n_steps; ++t) {
    if (t + 1 < n_steps) cp_async_wait<1>();
    else cp_async_wait<0>();
    __syncthreads();
    if (t == 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int r = warp * 16 + (lane & 15), c = kk * 2 + (lane >> 4);
        ldsm_x4(smem_u32(sQ) + swz(r, c), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
      cluster_arrive();  // this CTA's query staging is no longer read; its receive barrier is initialised
    }
    const int chunk = sub_of(t);
    uint8_t* stage = stage0 + (t & 1) * STAGE_BYTES;
#pragma unroll 1
    for (int sb = 0; sb < NSUB; ++sb) {
      const uint32_t kb = smem_u32(stage + sb * TILE_BYTES);
      const uint32_t vb = smem_u32(stage + (NSUB + sb) * TILE_BYTES);
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
      // mask (key position <= row position), scale to the log2 domain, online-softmax update
      const int kbase = chunk * kAttnChunk + sb * SUB + 2 * (lane & 3);
      float x_lo = -INFINITY, x_hi = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < SUB / 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int kp = kbase + nt * 8 + e;
          s[nt][e] = (kp <= pos_lo) ? s[nt][e] * a.scale_log2 : -INFINITY;
          s[nt][2 + e] = (kp <= pos_hi) ? s[nt][2 + e] * a.scale_log2 : -INFINITY;
          x_lo = fmaxf(x_lo, s[nt][e]);
          x_hi = fmaxf(x_hi, s[nt][2 + e]);
        }
      }
#pragma unroll
      for (int sh = 1; sh <= 2; sh <<= 1) {
        x_lo = fmaxf(x_lo, __shfl_xor_sync(0xffffffffu, x_lo, sh));
        x_hi = fmaxf(x_hi, __shfl_xor_sync(0xffffffffu, x_hi, sh));
      }
      const float mn_lo = fmaxf(m_lo, x_lo), mn_hi = fmaxf(m_hi, x_hi);
      const float al_lo = (m_lo == -INFINITY) ? 0.f : exp2f(m_lo - mn_lo);
      const float al_hi = (m_hi == -INFINITY) ? 0.f : exp2f(m_hi - mn_hi);
      const float b_lo = (mn_lo == -INFINITY) ? 0.f : mn_lo;
      const float b_hi = (mn_hi == -INFINITY) ? 0.f : mn_hi;
      m_lo = mn_lo;
      m_hi = mn_hi;
      l_lo *= al_lo;
      l_hi *= al_hi;
#pragma unroll
      for (int nt = 0; nt < SUB / 8; ++nt) {
        s[nt][0] = exp2f(s[nt][0] - b_lo);
        s[nt][1] = exp2f(s[nt][1] - b_lo);
        s[nt][2] = exp2f(s[nt][2] - b_hi);
        s[nt][3] = exp2f(s[nt][3] - b_hi);
        l_lo += s[nt][0] + s[nt][1];
        l_hi += s[nt][2] + s[nt][3];
      }
#pragma unroll
      for (int i = 0; i < HD / 8; ++i) {
        o[i][0] *= al_lo;
        o[i][1] *= al_lo;
        o[i][2] *= al_hi;
        o[i][3] *= al_hi;
      }
      // O += P V
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
    }
    __syncthreads();  // this stage is free again
    if (t + 2 < n_steps) {
      issue_kv(a, u, sub_of(t + 2), t + 2, max_kp, s_page, stage, 3);
      cp_async_commit();
    }
  }
  if (n_steps == 0) cluster_arrive();
#pragma unroll
  for (int sh = 1; sh <= 2; sh <<= 1) {
    l_lo += __shfl_xor_sync(0xffffffffu, l_lo, sh);
    l_hi += __shfl_xor_sync(0xffffffffu, l_hi, sh);
  }
  // this warp's lane state (rows 16w .. 16w+15) is staged as one block and copied into CTA w
  {
    float* blk = reinterpret_cast<float*>(stage0) + warp * BLOCK_FLOATS;  // stages are free after the loop
    const int d0 = 2 * (lane & 3);
    const int lr = lane >> 2;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      *reinterpret_cast<float2*>(blk + lr * HD + i * 8 + d0) = make_float2(o[i][0], o[i][1]);
      *reinterpret_cast<float2*>(blk + (lr + 8) * HD + i * 8 + d0) = make_float2(o[i][2], o[i][3]);
    }
    if ((lane & 3) == 0) {
      blk[ROWS_PER_CTA * HD + lr] = m_lo;
      blk[ROWS_PER_CTA * HD + lr + 8] = m_hi;
      blk[ROWS_PER_CTA * HD + ROWS_PER_CTA + lr] = l_lo;
      blk[ROWS_PER_CTA * HD + ROWS_PER_CTA + lr + 8] = l_hi;
    }
    fence_proxy_async_smem();  // make the block visible to the bulk-copy engine
    __syncwarp();
    if (tid == 0) mbar_arrive_expect_tx(smem_u32(&recv_bar), (uint32_t)RECV_BYTES);
    cluster_wait();  // every CTA of the cluster has its queries in registers: the receive buffers are free
    if (lane == 0) {
      const uint32_t peer = (uint32_t)warp;
      bulk_copy_to_cluster(dsmem_addr(smem_u32(recv + j * BLOCK_FLOATS), peer), smem_u32(blk), (uint32_t)BLOCK_BYTES,
                           dsmem_addr(smem_u32(&recv_bar), peer));
    }
  }
  // all 8 blocks of this CTA's rows have arrived
  const bool got = mbar_wait_cluster_bounded(smem_u32(&recv_bar), 0u, JF_WAIT_LIMIT_NS);
  if (!got && tid == 0) jf_set_error(a.err, JF_DERR_TIMEOUT_TMA);
  // fold of rows 16j .. 16j+15 over the 8 lanes in order; thread = (row, 8 of the 128 dims)
  {
    const int lr = tid >> 4, r = j * ROWS_PER_CTA + lr;
    const int d = (tid & 15) * 8;
    if (got && r < qrows) {
      const float* ro = recv + lr * HD + d;
      const float* rm = recv + ROWS_PER_CTA * HD + lr;
      const float* rl = rm + ROWS_PER_CTA;
      float M = rm[0], L = rl[0];
      float acc[8];
      {
        const float4 x0 = *reinterpret_cast<const float4*>(ro), x1 = *reinterpret_cast<const float4*>(ro + 4);
        acc[0] = x0.x; acc[1] = x0.y; acc[2] = x0.z; acc[3] = x0.w;
        acc[4] = x1.x; acc[5] = x1.y; acc[6] = x1.z; acc[7] = x1.w;
      }
#pragma unroll
      for (int q = 1; q < kAttnLanes; ++q) {
        float wa, wb, mm;
        fold_weights(M, rm[q * BLOCK_FLOATS], wa, wb, mm);
        const float4 x0 = *reinterpret_cast<const float4*>(ro + q * BLOCK_FLOATS);
        const float4 x1 = *reinterpret_cast<const float4*>(ro + q * BLOCK_FLOATS + 4);
        M = mm;
        L = wa * L + wb * rl[q * BLOCK_FLOATS];
        acc[0] = wa * acc[0] + wb * x0.x; acc[1] = wa * acc[1] + wb * x0.y;
        acc[2] = wa * acc[2] + wb * x0.z; acc[3] = wa * acc[3] + wb * x0.w;
        acc[4] = wa * acc[4] + wb * x1.x; acc[5] = wa * acc[5] + wb * x1.y;
        acc[6] = wa * acc[6] + wb * x1.z; acc[7] = wa * acc[7] + wb * x1.w;
      }
      const float il = L > 0.f ? 1.f / L : 0.f;
      const int qr = qr0 + r, t = qr / G, g = qr % G;
      bf16* dst = reinterpret_cast<bf16*>(a.out) + ((size_t)(u.row0 + t) * a.Hq + u.kvh * G + g) * HD + d;
      *reinterpret_cast<uint4*>(dst) = make_uint4(pack_bf16(acc[0] * il, acc[1] * il), pack_bf16(acc[2] * il, acc[3] * il),
                                                  pack_bf16(acc[4] * il, acc[5] * il), pack_bf16(acc[6] * il, acc[7] * il));
    }
  }
  // every copy out of this CTA's shared memory has landed (each CTA has received all it was sent)
  cluster_sync();
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

}  // namespace

size_t attn_bf16_smem_bytes() { return (size_t)ATT_SMEM; }

cudaError_t attn_prepare() {
  cudaError_t e = cudaFuncSetAttribute(k_attn_bf16, cudaFuncAttributeMaxDynamicSharedMemorySize, ATT_SMEM);
  if (e != cudaSuccess) return e;
  // an 8-CTA cluster of this kernel must fit on the device
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kAttnLanes);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = ATT_SMEM;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = kAttnLanes;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n_clusters = 0;
  e = cudaOccupancyMaxActiveClusters(&n_clusters, k_attn_bf16, &cfg);
  if (e != cudaSuccess) return e;
  return n_clusters > 0 ? cudaSuccess : cudaErrorInvalidConfiguration;
}

cudaError_t launch_attn_bf16(const AttnParams& a, int units_bound, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kAttnLanes * units_bound);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = ATT_SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = kAttnLanes;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, k_attn_bf16, a);
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
