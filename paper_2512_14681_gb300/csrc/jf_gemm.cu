// Weight-streaming projections of the forward pass (Eq. 3: one pass over all in-flight rows):
// Y[m, n] = sum_k X[m, k] W[n, k] for the QKV, O, gate/up, down and LM-head matrices.
//
// bf16 path: tcgen05 tensor cores, "swap-AB" so that 128 weight rows form the MMA's M side and
// the (few) in-flight tokens its N side. A persistent, warp-specialised kernel: one CTA per SM
// walks its share of (tile, split) work units; a producer warp streams weight and activation
// tiles by TMA (128-byte swizzle) through a 4-12 stage mbarrier ring that never drains between
// units; an MMA warp accumulates into one of two TMEM accumulators; four epilogue warps drain
// the other accumulator (fused epilogue, split-K reduction) while the next unit streams in.
// fp32 path (small fp32 models): a SIMT mainloop with the same tile shape and epilogues.
//
// Split-K is deterministic: partial tiles go to a workspace and the last CTA of a tile (atomic
// ticket, no waiting) adds them in split order. Every output element's reduction order is fixed
// by the weight shape alone, so a row's result does not depend on how many rows are in flight.
#include "jf_device.cuh"
#include "jf_internal.h"
#include "jf_once.h"

namespace jf {
namespace {

constexpr int A_STAGE_BYTES = kTileN * kTileK * 2;  // 16 KB of weights per stage

constexpr int EPI_STAGE_BYTES = 16 * kTileN * 4;   // epilogue exchange buffer [16][128] fp32
constexpr int SMEM_LIMIT = 232448;                  // 227 KB per CTA

template <int BN>
struct TcCfg {
  static constexpr int B_STAGE_BYTES = BN * kTileK * 2;
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr int S0 = (SMEM_LIMIT - 1024 - EPI_STAGE_BYTES - 512) / STAGE_BYTES;
  static constexpr int STAGES = S0 < 2 ? 2 : (S0 > 12 ? 12 : S0);
  static constexpr int ACC_COLS = BN;   // one accumulator; two are allocated (double buffer)
  static constexpr int TMEM_COLS = 2 * BN <= 32 ? 32 : (2 * BN <= 64 ? 64 : (2 * BN <= 128 ? 128 : (2 * BN <= 256 ? 256 : 512)));
  static constexpr int SMEM = 1024 + STAGES * STAGE_BYTES + EPI_STAGE_BYTES + 512;
  static_assert(SMEM <= SMEM_LIMIT, "shared memory budget");
};

// Named barrier of the 128 epilogue threads (barrier 0 is __syncthreads).
JF_DEV void epi_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

constexpr int kMaxSplits = 8;  // split-K never exceeds this (enforced by the host)

JF_DEV uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// ---------------------------------------------------------------------------------------------
// Epilogue on one 16-column chunk: thread `row` (0..127) holds v[j] = Y[m0 + c0 + j, n0 + row].
// xs: shared staging [16][128] fp32 (exchange between the two halves of a tile).
// ---------------------------------------------------------------------------------------------
template <typename T, int EPI>
JF_DEV void epilogue_chunk(const GemmEpi& e, const float (&v)[16], int row, int n0, int m0, int c0, float* xs,
                           int n_tile, int slot, int n_slots) {
  const int n = n0 + row;
  constexpr int kind = EPI;
  if constexpr (kind == EPI_STORE || kind == EPI_RESID) {
    if (n < e.N) {
      if constexpr (kind == EPI_RESID) {
        // all residual loads first (independent), then the stores
        float old[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int m = m0 + c0 + j;
          old[j] = (m < e.M) ? e.x[(size_t)m * e.ldx + n] : 0.0f;
        }
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int m = m0 + c0 + j;
          if (m < e.M) e.x[(size_t)m * e.ldx + n] = old[j] + v[j];
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int m = m0 + c0 + j;
          if (m < e.M) e.y[(size_t)m * e.ldy + n] = v[j];
        }
      }
    }
    return;
  } else if constexpr (kind == EPI_SWIGLU) {
    // rows 2i (gate) and 2i+1 (up) of the tile are feature 64 * n_tile + i, held by adjacent lanes:
    // the even lane finishes columns 0..7 of the chunk, the odd lane columns 8..15
    const bool odd = (row & 1) != 0;
    const int f = n_tile * 64 + (row >> 1);
    T* act = reinterpret_cast<T*>(e.act);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float mine = odd ? v[k] : v[8 + k];
      const float other = __shfl_xor_sync(0xffffffffu, mine, 1);
      const float g = odd ? other : v[k];
      const float u = odd ? v[8 + k] : other;
      const int m = m0 + c0 + (odd ? 8 + k : k);
      if (m < e.M && n < e.N) act[(size_t)m * e.ld_act + f] = to_act<T>(silu_f(g) * u);
    }
    return;
  } else if constexpr (kind == EPI_QKV) {
    // the feature's bias (if any) before the rotation, so that the partner reads biased values
    const float b = (e.bias != nullptr && n < e.N) ? act_to_f32(reinterpret_cast<const T*>(e.bias)[n]) : 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j) xs[j * 128 + row] = v[j] + b;
    epi_sync();
    {
      const int hd = e.head_dim, half = hd >> 1;
      const int i = n % hd;
      const bool is_q = n < e.n_q;
      const bool is_k = !is_q && n < e.n_q + e.n_kv;
      const bool rot = is_q || is_k;
      const int partner = (i < half) ? row + half : row - half;
      T* dst;
      size_t stride;
      if (is_q) { dst = reinterpret_cast<T*>(e.q_out) + n; stride = (size_t)e.n_q; }
      else if (is_k) { dst = reinterpret_cast<T*>(e.k_out) + (n - e.n_q); stride = (size_t)e.n_kv; }
      else { dst = reinterpret_cast<T*>(e.v_out) + (n - e.n_q - e.n_kv); stride = (size_t)e.n_kv; }
      if (n < e.N) {
        // positions, then rotary coefficients: two rounds of independent loads for 16 tokens
        int pm[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int m = m0 + c0 + j;
          pm[j] = (rot && m < e.M) ? e.pos[m] : 0;
        }
        float2 cs[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) cs[j] = rot ? e.rope[(size_t)pm[j] * half + (i % half)] : make_float2(1.f, 0.f);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int m = m0 + c0 + j;
          float out = xs[j * 128 + row];
          if (rot) {
            const float x2 = xs[j * 128 + partner];
            out = (i < half) ? (out * cs[j].x - x2 * cs[j].y) : (out * cs[j].x + x2 * cs[j].y);
          }
          if (m < e.M) dst[(size_t)m * stride] = to_act<T>(out);
        }
      }
    }
    epi_sync();
    return;
  } else {
    // EPI_ARGMAX: best (value, index) and runner-up value over this tile's 128 vocabulary rows
    float* red = xs;  // [4 warps][16 cols][3]
    const int warp = row >> 5, lane = row & 31;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float b1 = (n < e.N) ? v[j] : -INFINITY;
      int bi = (n < e.N) ? n : 0x7fffffff;
      float b2 = -INFINITY;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float o1 = __shfl_xor_sync(0xffffffffu, b1, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        const float o2 = __shfl_xor_sync(0xffffffffu, b2, o);
        if (better(o1, oi, b1, bi)) { b2 = fmaxf(b1, o2); b1 = o1; bi = oi; }
        else { b2 = fmaxf(b2, o1); }
      }
      if (lane == 0) {
        red[(warp * 16 + j) * 3 + 0] = b1;
        red[(warp * 16 + j) * 3 + 1] = __int_as_float(bi);
        red[(warp * 16 + j) * 3 + 2] = b2;
      }
    }
    epi_sync();
    if (row < 16) {
      const int j = row, m = m0 + c0 + j;
      float b1 = red[j * 3 + 0], b2 = red[j * 3 + 2];
      int bi = __float_as_int(red[j * 3 + 1]);
      for (int w = 1; w < 4; ++w) {
        const float o1 = red[(w * 16 + j) * 3 + 0], o2 = red[(w * 16 + j) * 3 + 2];
        const int oi = __float_as_int(red[(w * 16 + j) * 3 + 1]);
        if (better(o1, oi, b1, bi)) { b2 = fmaxf(b1, o2); b1 = o1; bi = oi; }
        else { b2 = fmaxf(b2, o1); }
      }
      if (m < e.M) {
        // fold this tile into the CTA's running (best, index, runner-up) of row m; the same
        // thread owns the slot for every tile of the CTA, so program order orders the updates
        const size_t at = (size_t)m * n_slots + slot;
        const float o1 = e.am_v1[at], o2 = e.am_v2[at];
        const int oi = e.am_i1[at];
        if (better(b1, bi, o1, oi)) {
          e.am_v1[at] = b1;
          e.am_i1[at] = bi;
          e.am_v2[at] = fmaxf(o1, b2);
        } else {
          e.am_v2[at] = fmaxf(o2, b1);
        }
      }
    }
    epi_sync();
  }
}

// Argmax partials: slot (m, s) holds CTA s's running (best value, its index, runner-up value) of
// row m over the vocabulary tiles that CTA has folded in. Every CTA starts its slots empty.
JF_DEV void argmax_init_slots(const GemmEpi& e, int m_begin, int m_end, int slot, int n_slots, int tid, int nthreads) {
  if (m_end > e.M) m_end = e.M;
  for (int m = m_begin + tid; m < m_end; m += nthreads) {
    const size_t at = (size_t)m * n_slots + slot;
    e.am_v1[at] = -INFINITY;
    e.am_i1[at] = 0x7fffffff;
    e.am_v2[at] = -INFINITY;
  }
}

JF_DEV void am_merge(float& b1, int& bi, float& b2, float o1, int oi, float o2) {
  if (better(o1, oi, b1, bi)) { b2 = fmaxf(b1, o2); b1 = o1; bi = oi; }
  else { b2 = fmaxf(b2, o1); }
}

// Last CTA of a token tile: reduce the slots of rows m0..m0+BN-1. Warp w takes rows two at a
// time, lane l the slots l, l+32, ...; each round issues all loads of 2 rows x 4 slots per lane
// before the first merge. The merge is associative and commutative, so the result does
// not depend on which CTA folded which tile.
constexpr int kAmSlotLoads = 4;  // slots per lane in flight per round
JF_DEV void argmax_finish(const GemmEpi& e, int m0, int BN, int n_slots, int tid) {
  const int warp = tid >> 5, lane = tid & 31;
  for (int r0 = warp * 2; r0 < BN; r0 += 8) {
    float b1[2] = {-INFINITY, -INFINITY}, b2[2] = {-INFINITY, -INFINITY};
    int bi[2] = {0x7fffffff, 0x7fffffff};
    for (int s0 = 0; s0 < n_slots; s0 += 32 * kAmSlotLoads) {
      float v1[2][kAmSlotLoads], v2[2][kAmSlotLoads];
      int i1[2][kAmSlotLoads];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const int m = m0 + r0 + q;
#pragma unroll
        for (int k = 0; k < kAmSlotLoads; ++k) {
          const int s = s0 + lane + 32 * k;
          const bool ok = (r0 + q < BN) && m < e.M && s < n_slots;
          const size_t at = (size_t)(ok ? m : 0) * n_slots + (ok ? s : 0);
          v1[q][k] = ok ? __ldcg(e.am_v1 + at) : -INFINITY;
          i1[q][k] = ok ? __ldcg(e.am_i1 + at) : 0x7fffffff;
          v2[q][k] = ok ? __ldcg(e.am_v2 + at) : -INFINITY;
        }
      }
#pragma unroll
      for (int q = 0; q < 2; ++q)
#pragma unroll
        for (int k = 0; k < kAmSlotLoads; ++k) am_merge(b1[q], bi[q], b2[q], v1[q][k], i1[q][k], v2[q][k]);
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int m = m0 + r0 + q;
      float b1q = b1[q], b2q = b2[q];
      int biq = bi[q];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float o1 = __shfl_xor_sync(0xffffffffu, b1q, o);
        const int oi = __shfl_xor_sync(0xffffffffu, biq, o);
        const float o2 = __shfl_xor_sync(0xffffffffu, b2q, o);
        am_merge(b1q, biq, b2q, o1, oi, o2);
      }
      if (lane == 0 && r0 + q < BN && m < e.M) {
        e.am_out[m] = biq;
        if (e.top2_out) { e.top2_out[2 * m] = b1q; e.top2_out[2 * m + 1] = b2q; }
      }
    }
  }
}

template <typename T, int BN, int EPI, typename Get>
JF_DEV void finish_tile_epi(const GemmParams& p, Get get, float* xs, int* sflag, int n_tile, int split, int m_tile,
                            int tid, int n0, int m0, int tile_lin, int nchunks);

// Shared tail of both mainloops, run by the 128 epilogue threads (tid 0..127): the partial tile
// for EPI_PARTIAL; otherwise ticketing for split-K and argmax, then the epilogue. get(c0, v) fills
// this thread's 16 accumulator values of columns c0..c0+15.
template <typename T, int BN, int EPI, typename Get>
JF_DEV void finish_tile(const GemmParams& p, Get get, float* xs, int* sflag, int n_tile, int split, int m_tile,
                        int tid) {
  const int n0 = n_tile * kTileN, m0 = m_tile * BN;
  const int tile_lin = n_tile * p.m_tiles + m_tile;
  int ncols = p.M - m0;
  if (ncols > BN) ncols = BN;
  const int nchunks = (ncols + 15) >> 4;
  if constexpr (EPI == EPI_PARTIAL) {
    float* mine = p.ws + ((size_t)tile_lin * p.k_splits + split) * (size_t)BN * kTileN;
    for (int c = 0; c < nchunks; ++c) {
      float v[16];
      get(c * 16, v);
#pragma unroll
      for (int j = 0; j < 16; ++j) mine[(c * 16 + j) * kTileN + tid] = v[j];
    }
  } else {
    finish_tile_epi<T, BN, EPI>(p, get, xs, sflag, n_tile, split, m_tile, tid, n0, m0, tile_lin, nchunks);
  }
}

template <typename T, int BN, int EPI, typename Get>
JF_DEV void finish_tile_epi(const GemmParams& p, Get get, float* xs, int* sflag, int n_tile, int split, int m_tile,
                            int tid, int n0, int m0, int tile_lin, int nchunks) {
  if (p.k_splits == 1) {
    for (int c = 0; c < nchunks; ++c) {
      float v[16];
      get(c * 16, v);
      epilogue_chunk<T, EPI>(p.epi, v, tid, n0, m0, c * 16, xs, n_tile, blockIdx.x, gridDim.x);
    }
  } else {
    float* mine = p.ws + ((size_t)tile_lin * p.k_splits + split) * (size_t)BN * kTileN;
    for (int c = 0; c < nchunks; ++c) {
      float v[16];
      get(c * 16, v);
#pragma unroll
      for (int j = 0; j < 16; ++j) mine[(c * 16 + j) * kTileN + tid] = v[j];
    }
    __threadfence();
    epi_sync();
    if (tid == 0) {
      const int t = atomicAdd(p.tile_counter + tile_lin, 1);
      *sflag = (t == p.k_splits - 1);
    }
    epi_sync();
    const bool last = *sflag != 0;
    epi_sync();
    if (!last) return;
    __threadfence();
    const float* base = p.ws + (size_t)tile_lin * p.k_splits * (size_t)BN * kTileN;
    for (int c = 0; c < nchunks; ++c) {
      // partials of every split in flight together, then added in split order
      float part[kMaxSplits][16];
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) {
        const float* src = base + (size_t)s * BN * kTileN;
#pragma unroll
        for (int j = 0; j < 16; ++j) part[s][j] = (s < p.k_splits) ? __ldcg(src + (c * 16 + j) * kTileN + tid) : 0.0f;
      }
      float v[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = 0.0f;
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) {
        if (s < p.k_splits) {
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] += part[s][j];
        }
      }
      epilogue_chunk<T, EPI>(p.epi, v, tid, n0, m0, c * 16, xs, n_tile, blockIdx.x, gridDim.x);
    }
    if (tid == 0) p.tile_counter[tile_lin] = 0;
  }
  if constexpr (EPI == EPI_ARGMAX) {
    __threadfence();
    epi_sync();
    if (tid == 0) {
      const int t = atomicAdd(p.epi.am_counter + m_tile, 1);
      *sflag = (t == p.n_tiles - 1);
    }
    epi_sync();
    const bool last = *sflag != 0;
    epi_sync();
    if (last) {
      __threadfence();
      argmax_finish(p.epi, m0, BN, gridDim.x, tid);
      if (tid == 0) p.epi.am_counter[m_tile] = 0;
    }
  }
}

// Work unit u of the persistent schedule: split = u % k_splits; the k_splits units of a tile are
// consecutive (their partials meet soon), and so are the m tiles of a weight tile (its second
// read hits L2).
struct Unit {
  int n_tile, m_tile, split, kb0, kb1;
};
JF_DEV Unit unit_of(const GemmParams& p, int u) {
  Unit w;
  w.split = u % p.k_splits;
  const int t = u / p.k_splits;
  w.m_tile = t % p.m_tiles;
  w.n_tile = t / p.m_tiles;
  w.kb0 = (int)(((long long)p.kb_total * w.split) / p.k_splits);
  w.kb1 = (int)(((long long)p.kb_total * (w.split + 1)) / p.k_splits);
  return w;
}

// ---------------------------------------------------------------------------------------------
// bf16 tcgen05 persistent kernel, 192 threads: warps 0-3 epilogue (warp w reads TMEM lanes
// 32w .. 32w+31), warp 4 lane 0 = TMA producer (warp 4 also owns the TMEM allocation),
// warp 5 lane 0 = MMA issuer.
// ---------------------------------------------------------------------------------------------
constexpr int TC_THREADS = 192;

JF_DEV void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

template <int BN, int EPI>
__global__ void __launch_bounds__(TC_THREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const GemmParams p) {
  using Cfg = TcCfg<BN>;
  constexpr int S = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * A_STAGE_BYTES;
  float* xs = reinterpret_cast<float*>(sB + S * Cfg::B_STAGE_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(xs) + EPI_STAGE_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 4);
  int* sflag = reinterpret_cast<int*>(tmem_slot + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + S);
  const uint32_t tfull0 = smem_u32(bars + 2 * S), tempty0 = smem_u32(bars + 2 * S + 2);
  const int total_units = p.n_tiles * p.m_tiles * p.k_splits;
  JF_TL_ENTRY();
  // The next kernel may launch as soon as every CTA of this grid is resident: its CTAs take the
  // SMs this grid leaves, prefetch their own weights and park in their dependency wait, so no
  // launch latency is paid after the last tile (it writes nothing before that wait).
  pdl_launch_dependents();

  // producer: initialise the barriers, then request the first weight stages right away (weights do
  // not depend on earlier kernels, so they stream in while the previous kernel finishes)
  int total_iters = 0;
  for (int u = blockIdx.x; u < total_units; u += gridDim.x) {
    const Unit w = unit_of(p, u);
    total_iters += w.kb1 - w.kb0;
  }
  const int pre = total_iters < S ? total_iters : S;
  if (tid == 128) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 1);
    }
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    const uint64_t polA = l2_policy_evict_first();
    int u = blockIdx.x, kb = 0;
    Unit w = unit_of(p, u);
    kb = w.kb0;
    for (int j = 0; j < pre; ++j) {
      mbar_arrive_expect_tx(full0 + 8 * j, Cfg::STAGE_BYTES);
      tma_load_2d(smem_u32(sA + j * A_STAGE_BYTES), &tmA, full0 + 8 * j, kb * kTileK, w.n_tile * kTileN, polA);
      if (++kb == w.kb1) {
        u += gridDim.x;
        if (u < total_units) {
          w = unit_of(p, u);
          kb = w.kb0;
        }
      }
    }
  }
  __syncwarp();
  if (warp == 4) {
    tmem_alloc(smem_u32(tmem_slot), Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 4) {
    if (lane == 0) {
      const uint64_t polA = l2_policy_evict_first(), polB = l2_policy_evict_last();
      pdl_wait();
      // activations of the prefetched stages
      {
        int u = blockIdx.x;
        Unit w = unit_of(p, u);
        int kb = w.kb0;
        for (int j = 0; j < pre; ++j) {
          tma_load_2d(smem_u32(sB + j * Cfg::B_STAGE_BYTES), &tmB, full0 + 8 * j, kb * kTileK, w.m_tile * BN, polB);
          if (++kb == w.kb1) {
            u += gridDim.x;
            if (u < total_units) {
              w = unit_of(p, u);
              kb = w.kb0;
            }
          }
        }
      }
      // steady state
      int j = 0;
      for (int u = blockIdx.x; u < total_units; u += gridDim.x) {
        const Unit w = unit_of(p, u);
        bool ok = true;
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++j) {
          if (j < pre) continue;
          const int s = j % S;
          if (!mbar_wait_bounded(empty0 + 8 * s, (uint32_t)((j / S) - 1) & 1u, p.wait_ns)) {
            jf_set_error(p.err, JF_DERR_TIMEOUT_MMA);
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full0 + 8 * s, Cfg::STAGE_BYTES);
          tma_load_2d(smem_u32(sA + s * A_STAGE_BYTES), &tmA, full0 + 8 * s, kb * kTileK, w.n_tile * kTileN, polA);
          tma_load_2d(smem_u32(sB + s * Cfg::B_STAGE_BYTES), &tmB, full0 + 8 * s, kb * kTileK, w.m_tile * BN, polB);
        }
        if (!ok) break;
      }
    }
  } else if (warp == 5) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kTileN, BN);
      int j = 0, i = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < total_units && ok; u += gridDim.x, ++i) {
        const Unit w = unit_of(p, u);
        const int acc = i & 1;
        if (i >= 2 && !mbar_wait_bounded(tempty0 + 8 * acc, (uint32_t)((i >> 1) - 1) & 1u, p.wait_ns)) {
          jf_set_error(p.err, JF_DERR_TIMEOUT_EPI);
          break;
        }
        tc_fence_after();
        const uint32_t dacc = tmem + (uint32_t)(acc * Cfg::ACC_COLS);
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++j) {
          const int s = j % S;
          if (!mbar_wait_bounded(full0 + 8 * s, (uint32_t)(j / S) & 1u, p.wait_ns)) {
            jf_set_error(p.err, JF_DERR_TIMEOUT_TMA);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a = smem_u32(sA + s * A_STAGE_BYTES), b = smem_u32(sB + s * Cfg::B_STAGE_BYTES);
#pragma unroll
          for (int kk = 0; kk < kTileK / 16; ++kk)
            tc_mma_bf16(dacc, sdesc_k_sw128(a + kk * 32), sdesc_k_sw128(b + kk * 32), idesc,
                        (kb > w.kb0 || kk > 0) ? 1u : 0u);
          tc_commit(empty0 + 8 * s);
        }
        tc_commit(tfull0 + 8 * acc);
      }
    }
  } else {
    // epilogue warps 0-3
    pdl_wait();
    JF_TL_WAITED();
    if constexpr (EPI == EPI_ARGMAX) {
      argmax_init_slots(p.epi, 0, p.M, blockIdx.x, gridDim.x, tid, 128);
      epi_sync();
    }
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    int i = 0;
    for (int u = blockIdx.x; u < total_units; u += gridDim.x, ++i) {
      const Unit w = unit_of(p, u);
      const int acc = i & 1;
      if (!mbar_wait_bounded(tfull0 + 8 * acc, (uint32_t)(i >> 1) & 1u, p.wait_ns)) {
        jf_set_error(p.err, JF_DERR_TIMEOUT_EPI);
        break;
      }
      tc_fence_after();
      const uint32_t dacc = tmem + (uint32_t)(acc * Cfg::ACC_COLS) + lane_base;
      auto get = [&](int c0, float (&v)[16]) { tmem_ld16(dacc + (uint32_t)c0, v); };
      finish_tile<bf16, BN, EPI>(p, get, xs, sflag, w.n_tile, w.split, w.m_tile, tid);
      tc_fence_before();
      epi_sync();
      if (tid == 0) mbar_arrive(tempty0 + 8 * acc);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 4) tmem_dealloc(tmem, Cfg::TMEM_COLS);
  JF_TL_EXIT(TL_GEMM + EPI);
}

// ---------------------------------------------------------------------------------------------
// fp32 SIMT kernel: thread `row` accumulates Y[m0 .. m0+31, n0 + row] over K in fp32, in
// increasing k, with the token tile staged in shared memory.
// ---------------------------------------------------------------------------------------------
constexpr int F32_BN = 32;
constexpr int F32_BK = 32;

template <int EPI>
__global__ void __launch_bounds__(128) k_gemm_f32(const float* __restrict__ W, const float* __restrict__ X,
                                                  const GemmParams p) {
  __shared__ float xt[F32_BN][F32_BK + 1];
  __shared__ float xs[16 * 128];
  __shared__ int sflag;
  const int tid = threadIdx.x;
  const int n0 = blockIdx.x * kTileN, m0 = blockIdx.z * F32_BN;
  const int n = n0 + tid;
  pdl_wait();
  float acc[F32_BN];
#pragma unroll
  for (int j = 0; j < F32_BN; ++j) acc[j] = 0.0f;
  for (int k0 = 0; k0 < p.K; k0 += F32_BK) {
    for (int i = tid; i < F32_BN * F32_BK; i += 128) {
      const int r = i / F32_BK, c = i % F32_BK;
      const int m = m0 + r, k = k0 + c;
      xt[r][c] = (m < p.M && k < p.K) ? X[(size_t)m * p.K + k] : 0.0f;
    }
    __syncthreads();
    if (n < p.N) {
      const float* wr = W + (size_t)n * p.K + k0;
      const int kmax = (p.K - k0) < F32_BK ? (p.K - k0) : F32_BK;
      for (int c = 0; c < kmax; ++c) {
        const float w = wr[c];
#pragma unroll
        for (int j = 0; j < F32_BN; ++j) acc[j] = fmaf(w, xt[j][c], acc[j]);
      }
    }
    __syncthreads();
  }
  pdl_launch_dependents();
  auto get = [&](int c0, float (&v)[16]) {
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = 0.0f;
#pragma unroll
    for (int cc = 0; cc < F32_BN; cc += 16)
      if (cc == c0) {
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = acc[cc + j];
      }
  };
  if constexpr (EPI == EPI_ARGMAX) {
    argmax_init_slots(p.epi, m0, m0 + F32_BN, blockIdx.x, gridDim.x, tid, 128);
    __syncthreads();
  }
  finish_tile<float, F32_BN, EPI>(p, get, xs, &sflag, blockIdx.x, 0, blockIdx.z, tid);
}

template <int BN, int EPI>
cudaError_t launch_tc_epi(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p, cudaStream_t st) {
  using Cfg = TcCfg<BN>;
  cudaLaunchConfig_t cfg = {};
  const int units = p.n_tiles * p.m_tiles * p.k_splits;
  cfg.gridDim = dim3(units < p.grid ? units : p.grid);
  cfg.blockDim = dim3(TC_THREADS);
  cfg.dynamicSmemBytes = Cfg::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_gemm_tc<BN, EPI>, tmA, tmB, p);
}

template <int BN>
cudaError_t launch_tc(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p, cudaStream_t st) {
  switch (p.epi.kind) {
    case EPI_STORE: return launch_tc_epi<BN, EPI_STORE>(tmA, tmB, p, st);
    case EPI_RESID: return launch_tc_epi<BN, EPI_RESID>(tmA, tmB, p, st);
    case EPI_QKV: return launch_tc_epi<BN, EPI_QKV>(tmA, tmB, p, st);
    case EPI_SWIGLU: return launch_tc_epi<BN, EPI_SWIGLU>(tmA, tmB, p, st);
    case EPI_ARGMAX: return launch_tc_epi<BN, EPI_ARGMAX>(tmA, tmB, p, st);
    case EPI_PARTIAL: return launch_tc_epi<BN, EPI_PARTIAL>(tmA, tmB, p, st);
    default: return cudaErrorInvalidValue;
  }
}

template <int BN>
cudaError_t prep_tc() {
  cudaError_t e;
  const int sm = TcCfg<BN>::SMEM;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<BN, EPI_STORE>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm))) return e;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<BN, EPI_RESID>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm))) return e;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<BN, EPI_QKV>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm))) return e;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<BN, EPI_SWIGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm))) return e;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<BN, EPI_ARGMAX>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm))) return e;
  return cudaFuncSetAttribute(k_gemm_tc<BN, EPI_PARTIAL>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
}

}  // namespace

#ifdef JF_TIMELINE
JF_TL_SETTER(tl_set_gemm)
#endif

// Opt the tcgen05 kernels into their dynamic shared-memory sizes on the current device.
static cudaError_t gemm_prepare_current() {
  cudaError_t e;
  if ((e = prep_tc<32>()) != cudaSuccess) return e;
  if ((e = prep_tc<64>()) != cudaSuccess) return e;
  if ((e = prep_tc<128>()) != cudaSuccess) return e;
  if ((e = prep_tc<160>()) != cudaSuccess) return e;
  return prep_tc<256>();
}

// The attributes are per device: set them once for each device the process uses (outside any
// stream capture), whichever entry point reaches that device first.
cudaError_t gemm_prepare() {
  static PerDeviceOnce once;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const int r = once.run(dev, [] { return gemm_prepare_current(); });
  return r < 0 ? cudaErrorInvalidDevice : static_cast<cudaError_t>(r);
}

// Token-tile width: the narrowest tile that holds every row, 32 at the least (a 16-wide tile
// streamed the same weights measurably slower). Above 256 rows the rows take as few tiles as 256-wide
// ones would (every extra tile is one more pass over the weights), and among the widths that give
// that count the narrowest (the tensor cores' work grows with the padded rows): 320 rows = 2 x 160,
// 384 = 2 x 256 (3 x 128 measured slower), 512 = 2 x 256.
int gemm_bn_for(int M) {
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128) return 128;
  if (M <= 160) return 160;
  if (M <= 256) return 256;
  const int tiles = (M + 255) / 256;
  for (int bn : {128, 160})
    if ((M + bn - 1) / bn == tiles) return bn;
  return 256;
}

size_t gemm_smem_bytes(int bn) {
  switch (bn) {
    case 32: return TcCfg<32>::SMEM;
    case 64: return TcCfg<64>::SMEM;
    case 128: return TcCfg<128>::SMEM;
    case 160: return TcCfg<160>::SMEM;
    default: return TcCfg<256>::SMEM;
  }
}

cudaError_t launch_gemm_bf16(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p, int bn,
                             cudaStream_t st) {
  switch (bn) {
    case 32: return launch_tc<32>(tmA, tmB, p, st);
    case 64: return launch_tc<64>(tmA, tmB, p, st);
    case 128: return launch_tc<128>(tmA, tmB, p, st);
    case 160: return launch_tc<160>(tmA, tmB, p, st);
    case 256: return launch_tc<256>(tmA, tmB, p, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm_f32(const float* W, const float* X, const GemmParams& p, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_tiles, 1, p.m_tiles);
  cfg.blockDim = dim3(128);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  switch (p.epi.kind) {
    case EPI_STORE: return cudaLaunchKernelEx(&cfg, k_gemm_f32<EPI_STORE>, W, X, p);
    case EPI_RESID: return cudaLaunchKernelEx(&cfg, k_gemm_f32<EPI_RESID>, W, X, p);
    case EPI_QKV: return cudaLaunchKernelEx(&cfg, k_gemm_f32<EPI_QKV>, W, X, p);
    case EPI_SWIGLU: return cudaLaunchKernelEx(&cfg, k_gemm_f32<EPI_SWIGLU>, W, X, p);
    case EPI_ARGMAX: return cudaLaunchKernelEx(&cfg, k_gemm_f32<EPI_ARGMAX>, W, X, p);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace jf
