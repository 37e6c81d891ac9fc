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
// bf16 path: split-KV flash decoding on the tcgen05 tensor cores with a fixed reduction tree.
// Work unit = (chain, KV head, tile of 128 (token, head) query rows). Key positions are cut into
// absolute 128-key chunks, and chunk c belongs to lane c mod 8. A unit runs on 8 CTAs (an 8-CTA
// cluster while all units' clusters fit on the GPU at once, independent CTAs beyond that):
// CTA j walks the chunks of lane j in increasing order with one online-softmax state per row:
// S = Q K^T into tensor memory, the softmax step read straight out of it, P (fp16) back to shared
// memory, P V (fp16 operands; the cache holds V in fp16) into a second tensor-memory accumulator
// added into registers. K/V rows are staged by cp.async (the next chunk in flight while the
// current one computes). Each CTA then writes its
// lane state (O, running max, sum) to a global scratch slot of the unit; after a cluster barrier
// CTA j folds rows 16j .. 16j+15 over the 8 lanes in lane order (unclustered: the last lane to
// finish folds all rows, in the same order). The tree depends only on
// absolute key positions, never on how many rows share the forward or how many chunks a unit
// has, so a row's result is the same in every batch.
// fp32 path: one warp per (row, head), keys in absolute order, online softmax in fp32.
#include "jf_device.cuh"
#include "jf_internal.h"

namespace jf {
namespace {

constexpr int HD = 128;
constexpr int ROWS_PER_CTA = kAttnQRows / kAttnLanes;  // rows each CTA of a cluster folds (16)

JF_DEV void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}
JF_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
JF_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

JF_DEV uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);  // one cvt.rn.bf16x2.f32
  return *reinterpret_cast<const uint32_t*>(&v);
}

JF_DEV uint32_t pack_f16(float lo, float hi) {
  const __half2 v = __floats2half2_rn(lo, hi);  // one cvt.rn.f16x2.f32
  return *reinterpret_cast<const uint32_t*>(&v);
}

// 2^x by the MUFU ex2 instruction (flushes results below 2^-126 to zero; 2^-inf = 0).
JF_DEV float ex2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Fold of two softmax states (m, l, O) in the log2 domain: m = max(ma, mb),
// O = 2^(ma-m) Oa + 2^(mb-m) Ob, l likewise; an empty state has m = -inf and weight 0.
JF_DEV void fold_weights(float ma, float mb, float& wa, float& wb, float& m) {
  m = fmaxf(ma, mb);
  wa = (ma == -INFINITY) ? 0.f : exp2f(ma - m);
  wb = (mb == -INFINITY) ? 0.f : exp2f(mb - m);
}

// Unit ui of the forward (chains in order, then KV heads, then 128-row query tiles), looked up
// by warp 0 into s_unit; s_unit.pad stays 0 past the last unit. Every CTA of cluster ui gets the
// same unit. The chain table was written by host copies or an earlier graph launch, complete
// before this forward began, so this runs before the dependency wait.
JF_DEV void resolve_unit(const AttnParams& a, int ui, int j, int G, int warp, int lane, AttnUnit& s_unit) {
  if (threadIdx.x == 0) s_unit.pad = 0;
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
}

constexpr int ATT_THREADS = 256;

// ---------------------------------------------------------------------------------------------
// Per 128-key chunk of its lane a CTA computes S = Q K^T into TMEM (M = 128 query rows, N = 128
// keys, K = 128), takes the online-softmax step on S straight out of TMEM (warp w reads TMEM lanes
// 32(w%4).. and key columns 64(w/4)..+63; the two column halves of a row exchange their maxima in
// shared memory), writes P in fp16 as the next MMA's A operand and computes P V into a second TMEM
// accumulator, which the threads add into their registers (O = alpha O + P V). Every operand
// arrives as [key or row][128] in two 64-column blocks with the 128-byte swizzle: Q, K and P are
// read K-major, V (fp16 in the cache: the QKV finish stores the bf16-rounded values as fp16)
// MN-major as it arrives, dims along N. Q K^T runs on bf16 operands, P V on fp16 ones (both
// operands of one MMA share their type).
// ---------------------------------------------------------------------------------------------
constexpr int TC_BLK = 16384;                     // one 128-row x 64-column bf16 operand block
constexpr int TC_OPND = 2 * TC_BLK;               // 128 rows x 128 columns
constexpr int TC_OFF_Q = 0;
constexpr int TC_OFF_STAGE = TC_OPND;             // two stages of {K, V}
constexpr int TC_STAGE = 2 * TC_OPND;
constexpr int TC_SMEM = TC_OFF_STAGE + 2 * TC_STAGE + 1024;  // + slack for 1024-byte alignment
constexpr int TC_TMEM_COLS = 256;                 // S: columns 0..127, P V: columns 128..255

// byte offset of 16-byte chunk c16 (0..15) of row r in a [128][128] bf16 operand
JF_DEV uint32_t tc_swz(int r, int c16) {
  return (uint32_t)((c16 >> 3) * TC_BLK + r * 128 + (((c16 & 7) ^ (r & 7)) << 4));
}

// K and V rows of `chunk` into one stage ({K, V} in the operand layout); `part` selects the
// cached (1) and / or in-flight (2) keys.
JF_DEV void issue_kv_tc(const AttnParams& a, const AttnUnit& u, int chunk, int li, int max_kp, const int* s_page,
                        uint32_t stage, int part) {
  const bf16* Kp = reinterpret_cast<const bf16*>(a.k_pages);
  const __half* Vp = reinterpret_cast<const __half*>(a.v_pages);  // V is stored in fp16
  const bf16* Ki = reinterpret_cast<const bf16*>(a.k_inf);
  const __half* Vi = reinterpret_cast<const __half*>(a.v_inf);
  const int kp0 = chunk * kAttnChunk;
  for (int i = threadIdx.x; i < kAttnChunk * 16; i += blockDim.x) {
    const int r = i >> 4, c = i & 15;
    const int kp = kp0 + r;
    const bool cached = kp < u.pos0;
    if (!(part & (cached ? 1 : 2))) continue;
    const bf16* kr = nullptr;
    const __half* vr = nullptr;
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
    const uint32_t o = tc_swz(r, c);
    cp_async16(stage + o, kr ? kr + c * 8 : Kp, kr != nullptr);
    cp_async16(stage + TC_OPND + o, vr ? vr + c * 8 : Vp, vr != nullptr);
  }
}

// Fold of rows rb*16 .. rb*16+15 of unit ui over its 8 lane states in lane order (thread: row
// tid % 16, dims 8 (tid / 16) ..), normalised and stored in bf16. The same arithmetic whichever CTA
// of the unit runs it.
JF_DEV void fold_row_block(const AttnParams& a, const AttnUnit& u, int ui, int rb, int qr0, int qrows, int G, int tid) {
  const int lr = tid & 15, rw = rb * ROWS_PER_CTA + lr;
  const int d = (tid >> 4) * 8;
  if (rw >= qrows) return;
  const float* x0 = a.xchg + (size_t)ui * kAttnLanes * kAttnXchgFloats;
  float ov[kAttnLanes][8], mv[kAttnLanes], lv[kAttnLanes];
#pragma unroll
  for (int q = 0; q < kAttnLanes; ++q) {
    const float* xq = x0 + (size_t)q * kAttnXchgFloats;
#pragma unroll
    for (int e = 0; e < 8; ++e) ov[q][e] = __ldcg(xq + (d + e) * kAttnQRows + rw);
    mv[q] = __ldcg(xq + HD * kAttnQRows + rw);
    lv[q] = __ldcg(xq + HD * kAttnQRows + kAttnQRows + rw);
  }
  float M = mv[0], L = lv[0];
  float acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = ov[0][e];
#pragma unroll
  for (int q = 1; q < kAttnLanes; ++q) {
    float wa, wb, mm;
    fold_weights(M, mv[q], wa, wb, mm);
    M = mm;
    L = wa * L + wb * lv[q];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = wa * acc[e] + wb * ov[q][e];
  }
  const float il = L > 0.f ? 1.f / L : 0.f;
  const int qr = qr0 + rw, tq = qr / G, g = qr % G;
  bf16* dst = reinterpret_cast<bf16*>(a.out) + ((size_t)(u.row0 + tq) * a.Hq + u.kvh * G + g) * HD + d;
  *reinterpret_cast<uint4*>(dst) = make_uint4(pack_bf16(acc[0] * il, acc[1] * il), pack_bf16(acc[2] * il, acc[3] * il),
                                              pack_bf16(acc[4] * il, acc[5] * il), pack_bf16(acc[6] * il, acc[7] * il));
}

// kCluster: a unit's 8 lanes run as one 8-CTA cluster and, after a cluster barrier, CTA j folds
// rows 16j .. 16j+15 (the fastest fold; at most 15 such clusters of this kernel are resident on the
// 152 SMs at once). Otherwise the lanes are independent CTAs (all SMs usable) and the last lane of
// a unit to finish, found by a per-unit ticket, folds all 128 rows and resets the ticket. Both
// forms fold in lane order with the same arithmetic, so their results are bit-identical.
// At most 200 registers a thread, like the mma.sync kernel, so that its clusters are placed while
// the QKV finish kernel's CTAs are still resident.
template <bool kCluster>
__global__ void __maxnreg__(200) k_attn_tc(const AttnParams a) {
  extern __shared__ uint8_t sm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sQ = smem_u32(sm + TC_OFF_Q), sStage = smem_u32(sm + TC_OFF_STAGE);
  __shared__ __align__(8) uint64_t bars[2];                   // S ready, P V ready
  __shared__ uint32_t tmem_slot;
  __shared__ int s_rowpos[kAttnQRows];
  __shared__ int s_page[kAttnLaneChunks * (kAttnChunk / kPage)];
  __shared__ AttnUnit s_unit;
  __shared__ float red_max[2][kAttnQRows];
  __shared__ float red_l[2][kAttnQRows];
  __shared__ int s_last;

  JF_TL_ENTRY();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int j = (int)(blockIdx.x % kAttnLanes);  // = rank in the cluster when clustered
  const int ui = (int)(blockIdx.x / kAttnLanes);
  const int G = a.Hq / a.Hkv;
  const uint32_t s_full = smem_u32(&bars[0]), o_full = smem_u32(&bars[1]);
  pdl_launch_dependents();  // the next kernel may launch now
  if (tid == 0) {
    mbar_init(s_full, 1);
    mbar_init(o_full, 1);
    fence_mbar_init();
  }
  resolve_unit(a, ui, j, G, warp, lane, s_unit);
  const AttnUnit u = s_unit;
  if (!u.pad) return;  // past the last unit: the whole unit (cluster) leaves together
  if (warp == 0) {
    tmem_alloc(smem_u32(&tmem_slot), TC_TMEM_COLS);
    tmem_relinquish();
  }
  const int qr0 = u.qt * kAttnQRows;
  int qrows = u.nrows * G - qr0;
  if (qrows > kAttnQRows) qrows = kAttnQRows;
  const int max_kp = u.pos0 + (qr0 + qrows - 1) / G;
  const int n_steps = (u.n_chunks > j) ? (u.n_chunks - 1 - j) / kAttnLanes + 1 : 0;
  auto sub_of = [&](int t) { return j + kAttnLanes * t; };
  for (int i = tid; i < kAttnQRows; i += ATT_THREADS) s_rowpos[i] = (i < qrows) ? u.pos0 + (qr0 + i) / G : -1;
  for (int i = tid; i < n_steps * (kAttnChunk / kPage); i += ATT_THREADS) {
    const int li = i / (kAttnChunk / kPage), pg = i % (kAttnChunk / kPage);
    const int kp = (j + li * kAttnLanes) * kAttnChunk + pg * kPage;
    s_page[i] = (kp < u.pos0) ? a.page_table[(size_t)u.seq * a.pages_per_seq + (kp >> 4)] : -1;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  if (n_steps > 0) {
    issue_kv_tc(a, u, sub_of(0), 0, max_kp, s_page, sStage, 1);
    cp_async_commit();
  }
  pdl_wait();  // queries and in-flight keys come from the QKV projection
  JF_TL_WAITED();
  if (n_steps > 0) {
    const bf16* Q = reinterpret_cast<const bf16*>(a.q);
    for (int i = tid; i < kAttnQRows * 16; i += ATT_THREADS) {
      const int r = i >> 4, c = i & 15;
      const bool ok = r < qrows;
      const int qr = qr0 + (ok ? r : 0);
      const int t = qr / G, g = qr % G;
      const bf16* src = Q + ((size_t)(u.row0 + t) * a.Hq + u.kvh * G + g) * HD + c * 8;
      cp_async16(sQ + tc_swz(r, c), src, ok);
    }
    issue_kv_tc(a, u, sub_of(0), 0, max_kp, s_page, sStage, 2);
    cp_async_commit();
    if (n_steps > 1) {
      issue_kv_tc(a, u, sub_of(1), 1, max_kp, s_page, sStage + TC_STAGE, 3);
      cp_async_commit();
    }
  }

  const int quad = warp & 3, half = warp >> 2;
  const int r = quad * 32 + lane;  // this thread's query row (TMEM lane)
  const int pos_r = s_rowpos[r];
  const uint32_t t_row = tmem + ((uint32_t)(quad * 32) << 16);
  constexpr uint32_t idesc = idesc_bf16_f32(128, 128);
  constexpr uint32_t idesc_pv = idesc_f16_f32(128, 128) | (1u << 16);  // P V: fp16 P, fp16 V MN-major
  float o[64];
#pragma unroll
  for (int i = 0; i < 64; ++i) o[i] = 0.f;
  float m_run = -INFINITY, l_run = 0.f;
  bool ok = true;

  for (int t = 0; t < n_steps && ok; ++t) {
    if (t + 1 < n_steps) cp_async_wait<1>();
    else cp_async_wait<0>();
    const uint32_t sK = sStage + (uint32_t)((t & 1) * TC_STAGE), sV = sK + TC_OPND;
    fence_proxy_async_smem();  // this thread's cp.async writes -> tensor-core operand reads
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t off = (uint32_t)((kk >> 2) * TC_BLK + (kk & 3) * 32);
        tc_mma_bf16(tmem, sdesc_k_sw128(sQ + off), sdesc_k_sw128(sK + off), idesc, kk > 0 ? 1u : 0u);
      }
      tc_commit(s_full);
    }
    if (!mbar_wait_bounded(s_full, (uint32_t)(t & 1), a.wait_ns)) {
      if (tid == 0) jf_set_error(a.err, JF_DERR_TIMEOUT_MMA);
      ok = false;
    }
    tc_fence_after();
    // scores of this row, keys 64*half .. 64*half+63 of the chunk: mask, scale, row maximum
    float sv[64];
    {
      float t32[32];
      tmem_ld32(t_row + 64 * half, t32);
#pragma unroll
      for (int i = 0; i < 32; ++i) sv[i] = t32[i];
      tmem_ld32(t_row + 64 * half + 32, t32);
#pragma unroll
      for (int i = 0; i < 32; ++i) sv[32 + i] = t32[i];
    }
    const int kbase = sub_of(t) * kAttnChunk + 64 * half;
    // mask (key position <= row position) on the raw scores; the scale (> 0) goes into the row
    // maximum and into one fma per exponential: p = 2^(s * scale - m)
    const float scale = a.scale_log2;
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < 64; ++i) {
      sv[i] = (kbase + i <= pos_r) ? sv[i] : -INFINITY;
      mx = fmaxf(mx, sv[i]);
    }
    red_max[half][r] = mx * scale;
    ok = __syncthreads_and(ok) != 0;  // keeps the loop's barriers uniform across the CTA
    const float mn = fmaxf(m_run, fmaxf(red_max[0][r], red_max[1][r]));
    const float al = (m_run == -INFINITY) ? 0.f : ex2_ftz(m_run - mn);
    const float nb = (mn == -INFINITY) ? 0.f : -mn;
    m_run = mn;
    // P in fp16 into this stage's K block `half` (S is complete, K is no longer read): fp16 keeps
    // 11 significant bits of P in [0, 1], where bf16's 8 would move the attention output by up to
    // half a bf16 unit, as much as its own rounding. The row sum in four independent partial sums,
    // added in a fixed order.
    float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      float p[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        p[e] = ex2_ftz(fmaf(sv[8 * c + e], scale, nb));
        ls[e & 3] += p[e];
      }
      const uint4 w = make_uint4(pack_f16(p[0], p[1]), pack_f16(p[2], p[3]), pack_f16(p[4], p[5]),
                                 pack_f16(p[6], p[7]));
      const uint32_t dst = sK + (uint32_t)(half * TC_BLK + r * 128 + ((c ^ (r & 7)) << 4));
      asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(w.x), "r"(w.y), "r"(w.z), "r"(w.w)
                   : "memory");
    }
    l_run = l_run * al + ((ls[0] + ls[1]) + (ls[2] + ls[3]));
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t off = (uint32_t)((kk >> 2) * TC_BLK + (kk & 3) * 32);
        // keys 16kk .. 16kk+15 of V: 16 rows of 128 bytes; the two 64-dim atoms are a block apart
        tc_mma_bf16(tmem + 128, sdesc_k_sw128(sK + off), sdesc_mn_sw128(sV + (uint32_t)kk * 2048u, TC_BLK),
                    idesc_pv, kk > 0 ? 1u : 0u);
      }
      tc_commit(o_full);
    }
    if (!mbar_wait_bounded(o_full, (uint32_t)(t & 1), a.wait_ns)) {
      if (tid == 0) jf_set_error(a.err, JF_DERR_TIMEOUT_MMA);
      ok = false;
    }
    tc_fence_after();
    {
      float t32[32];
      tmem_ld32(t_row + 128 + 64 * half, t32);
#pragma unroll
      for (int i = 0; i < 32; ++i) o[i] = o[i] * al + t32[i];
      tmem_ld32(t_row + 128 + 64 * half + 32, t32);
#pragma unroll
      for (int i = 0; i < 32; ++i) o[32 + i] = o[32 + i] * al + t32[i];
    }
    tc_fence_before();
    ok = __syncthreads_and(ok) != 0;  // the stage and both TMEM accumulators are free again
    if (t + 2 < n_steps) {
      issue_kv_tc(a, u, sub_of(t + 2), t + 2, max_kp, s_page, sK, 3);
      cp_async_commit();
    }
  }
  cp_async_wait<0>();
  // lane state of the 128 rows (O, m, l over both column halves) to this lane's slot of the
  // unit in global memory, O stored dimension-major ([dim][row]: a warp writes 128 contiguous
  // bytes per dimension); then the fold (CTA j: rows 16j .. 16j+15 after the cluster barrier, or
  // the unit's last lane: all rows).
  red_l[half][r] = l_run;
  __syncthreads();
  float* xs = a.xchg + ((size_t)ui * kAttnLanes + j) * kAttnXchgFloats;
#pragma unroll
  for (int i = 0; i < 64; ++i) xs[(64 * half + i) * kAttnQRows + r] = o[i];
  if (half == 0) {
    xs[HD * kAttnQRows + r] = m_run;
    xs[HD * kAttnQRows + kAttnQRows + r] = red_l[0][r] + red_l[1][r];
  }
  if constexpr (kCluster) {
    cluster_sync();  // release / acquire: every lane's state of the unit is visible
    if (ok) fold_row_block(a, u, ui, j, qr0, qrows, G, tid);
  } else {
    __threadfence();  // this lane's state, then its ticket
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(a.unit_ticket + ui, 1) == kAttnLanes - 1;
    __syncthreads();
    if (s_last) {
      __threadfence();  // the other lanes' states are visible to the last one
      if (ok)
        for (int rb = 0; rb < kAttnLanes; ++rb) fold_row_block(a, u, ui, rb, qr0, qrows, G, tid);
      if (tid == 0) a.unit_ticket[ui] = 0;  // ready for the next launch
    }
  }
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, TC_TMEM_COLS);
  JF_TL_EXIT(TL_ATTN);
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
    if (kp <= pos) {
      if (kp < ch.pos0) {
        const int page = a.page_table[(size_t)ch.seq * a.pages_per_seq + (kp >> 4)];
        const size_t off = (((size_t)page * a.Hkv + kvh) * kPage + (kp & 15)) * hd;
        kr = Kp + off;
      } else {
        const size_t off = ((size_t)(ch.row0 + kp - ch.pos0) * a.Hkv + kvh) * hd;
        kr = Ki + off;
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
  }
  float* out = reinterpret_cast<float*>(a.out) + ((size_t)r * a.Hq + h) * hd;
  const float il = l > 0.f ? 1.f / l : 0.f;
  out[lane] = o0 * il;
  if (lane + 32 < hd) out[lane + 32] = o1 * il;
}

}  // namespace

#ifdef JF_TIMELINE
JF_TL_SETTER(tl_set_attn)
#endif

cudaError_t launch_attn_tc(const AttnParams& a, int units_bound, bool clustered, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kAttnLanes * units_bound);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = TC_SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = kAttnLanes;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = clustered ? 2 : 1;
  return clustered ? cudaLaunchKernelEx(&cfg, k_attn_tc<true>, a) : cudaLaunchKernelEx(&cfg, k_attn_tc<false>, a);
}

// Shared-memory limits of both forms; *max_clusters = how many 8-CTA clusters of the clustered
// form can be resident at once (0 = none, an error).
cudaError_t attn_prepare(int* max_clusters) {
  cudaError_t e = cudaFuncSetAttribute(k_attn_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_attn_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM);
  if (e != cudaSuccess) return e;
  // an 8-CTA cluster of this kernel must fit on the device
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kAttnLanes);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = TC_SMEM;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = kAttnLanes;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n_clusters = 0;
  e = cudaOccupancyMaxActiveClusters(&n_clusters, k_attn_tc<true>, &cfg);
  if (e != cudaSuccess) return e;
  *max_clusters = n_clusters;
  return n_clusters > 0 ? cudaSuccess : cudaErrorInvalidConfiguration;
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
