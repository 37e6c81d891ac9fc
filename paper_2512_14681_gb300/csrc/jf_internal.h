// Internal structures shared by the libjf host runtime and its kernels (not part of the C ABI).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace jf {

// Device error codes written into the context's error word (first writer wins).
enum DeviceError : int {
  JF_DERR_NONE = 0,
  JF_DERR_TIMEOUT_TMA = 1,   // a TMA transfer never completed its mbarrier
  JF_DERR_TIMEOUT_MMA = 2,   // an MMA commit never arrived
  JF_DERR_TIMEOUT_EPI = 3,   // the accumulator barrier never completed
  JF_DERR_BOUNDS = 4,        // a page-table / token / position index was out of range
  JF_DERR_STATE = 5,         // inconsistent decode state detected on the device
  JF_DERR_TIMEOUT_PROBE = 6, // the wait-limit probe's wait ran out (its intended outcome)
};

// Default limit of every bounded device wait: far beyond any legitimate wait. A context's limit
// is host-settable within [kWaitLimitMinNs, kWaitLimitMaxNs].
constexpr unsigned long long kWaitLimitDefaultNs = 2000000000ull;  // 2 s
constexpr unsigned long long kWaitLimitMinNs = 1000000ull;         // 1 ms
constexpr unsigned long long kWaitLimitMaxNs = 60000000000ull;     // 60 s


constexpr int kPage = 16;         // tokens per KV page
constexpr int kTileN = 128;       // weight rows per GEMM tile (tcgen05 M)
constexpr int kTileK = 64;        // K elements per GEMM pipeline stage
constexpr int kAttnChunk = 128;   // keys per split-KV chunk, aligned to absolute positions
constexpr int kAttnQRows = 128;   // (token, head) query rows per attention work unit
constexpr int kAttnLanes = 8;     // chunk lanes per unit (c mod 8); one CTA of an 8-CTA cluster each
constexpr int kAttnLaneChunks = 128;  // chunks per lane the kernel can stage page ids for
constexpr int kAttnMaxCtx = kAttnChunk * kAttnLanes * kAttnLaneChunks;  // 131072 key positions
constexpr int kAttnXchgFloats = kAttnQRows * 128 + 2 * kAttnQRows;   // one lane state: O (hd 128), m, l
constexpr int kMaxSeqs = 64;
constexpr int kMaxChains = 256;

// A chain: in-flight rows row0 .. row0+nrows-1 of sequence `seq` at consecutive positions
// pos0 .. pos0+nrows-1, where pos0 equals the sequence's committed length. Each row attends to
// the whole committed cache and to the rows of its own chain at positions <= its own.
struct Chain {
  int seq, row0, nrows, pos0;
};

// Attention work unit: (chain, KV head, tile of 128 (token, head) query rows), its chain resolved;
// `pad` is nonzero for a unit that exists.
struct AttnUnit {
  int seq, row0, nrows, pos0, kvh, qt, n_chunks, pad;
};

// EPI_PARTIAL: the tile's (split's) fp32 partial sums go to the workspace and the consumer kernel
// adds the k_splits partials of an element in split order (no ticket, no last-CTA reduction).
enum EpiKind : int { EPI_STORE = 0, EPI_RESID = 1, EPI_QKV = 2, EPI_SWIGLU = 3, EPI_ARGMAX = 4, EPI_PARTIAL = 5 };

// Where the consumer of an EPI_PARTIAL projection finds element (m, n): partial s lives at
// ws[((n / 128 * m_tiles + m / bn) * k_splits + s) * bn * 128 + (m % bn) * 128 + n % 128].
struct SplitPartials {
  const float* ws;
  int k_splits, m_tiles, bn;
};

struct GemmEpi {
  int kind;
  int M, N;
  // EPI_STORE: y[m * ldy + n] = v (fp32)
  float* y;
  int ldy;
  // EPI_RESID: x[m * ldx + n] += v (fp32 residual stream)
  float* x;
  int ldx;
  // EPI_QKV: rotary embedding on q/k features, then q -> q_out[m][Hq][hd], k/v -> k_out/v_out[m][Hkv][hd]
  void* q_out;
  void* k_out;
  void* v_out;
  int n_q, n_kv, head_dim;
  const int* pos;
  const float2* rope;   // [max_pos][hd/2] (cos, sin)
  const void* bias;     // per-feature Q/K/V biases [n_q + 2 n_kv] in the model dtype, added before RoPE, or null
  // EPI_SWIGLU: tile t holds features 64t..64t+63 as row pairs (gate 64t+i at 2i, up at 2i+1); act[m][64t + i]
  void* act;
  int ld_act;
  // EPI_ARGMAX: per (row, CTA) running (v1, i1, v2) slot, one ticket per token tile; the CTA that
  // completes a token tile folds the slots into the final argmax / top-2
  float* am_v1;
  int* am_i1;
  float* am_v2;
  int* am_counter;
  int* am_out;
  float* top2_out;
};

struct GemmParams {
  int N, K, M;
  int n_tiles, m_tiles, k_splits, kb_total;
  int grid;            // persistent CTAs (bf16 path): at most one per SM
  float* ws;           // split-K partials [n_tiles][m_tiles][k_splits][BN][128]
  int* tile_counter;   // [m_tiles*n_tiles], zero between launches
  int* err;
  unsigned long long wait_ns;  // limit of each bounded wait
  GemmEpi epi;
};

struct AttnParams {
  const void* q;        // [R][Hq][hd]
  const void* k_inf;    // this layer's in-flight K [R][Hkv][hd]
  const void* v_inf;
  const void* k_pages;  // this layer's K pages [n_pages][Hkv][16][hd]
  const void* v_pages;
  const int* page_table;  // [max_seqs][pages_per_seq]
  int pages_per_seq;
  int n_pages;
  const int* seq_len;   // committed length per sequence
  const Chain* chains;
  const int* n_chains_dev;
  void* out;            // [R][Hq*hd]
  int Hq, Hkv, hd;
  float scale_log2;     // log2(e) / sqrt(hd)
  int* err;
  unsigned long long wait_ns;  // limit of each bounded wait
  float* xchg;          // bf16 path: lane states [unit][lane][kAttnXchgFloats]
  int* unit_ticket;     // bf16 path, unclustered form: lanes finished per unit, zero between launches
};

// Host-side launch helpers of the projection GEMM (jf_gemm.cu) and the TMA descriptor encoder
// (jf_runtime.cu). All launches use programmatic dependent launch.
cudaError_t launch_gemm_bf16(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p, int bn,
                             cudaStream_t st);
cudaError_t launch_gemm_f32(const float* W, const float* X, const GemmParams& p, cudaStream_t st);
int gemm_bn_for(int M);
#ifdef JF_TIMELINE
// Timeline builds: point each translation unit's record buffer / counter at caller memory.
cudaError_t tl_set_gemm(void* records, void* counter);
cudaError_t tl_set_attn(void* records, void* counter);
cudaError_t tl_set_elem(void* records, void* counter);
cudaError_t tl_set_decode(void* records, void* counter);
#endif
size_t gemm_smem_bytes(int bn);
int gemm_default_splits(int n_tiles, int kb_total);
bool encode_tmap_bf16(CUtensorMap* tm, const void* ptr, long long K, long long rows, int box_rows);

}  // namespace jf
