// Host runtime of libjf: context and arena, weights, KV-page allocator, forward-pass launch
// sequence, CUDA graphs of the decode iteration, and the C ABI of include/jf.h / jf_ops.h.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstddef>
#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "../../include/jf.h"
#include "../../include/jf_ops.h"
#include "jf_attn_form.h"
#include "jf_decode.h"
#include "jf_internal.h"

namespace jf {
// kernels defined in the other translation units
cudaError_t launch_init_weights(void* dst, bool is_bf16, long long rows, long long cols, uint64_t seed, uint64_t tid,
                                double stdv, long long grp, long long grp_stride, long long grp_off, cudaStream_t st);
cudaError_t launch_fill_f32(float* p, long long n, float v, cudaStream_t st);
cudaError_t launch_rope_table(float2* tab, int n_pos, int half, double theta, cudaStream_t st);
cudaError_t launch_embed(const void* E, bool is_bf16, const int* tok, float* x, int rows, int d, int V, int* err,
                         cudaStream_t st);
cudaError_t launch_rmsnorm(float* x, const float* gain, void* y, bool is_bf16, int rows, int d, float eps,
                           const SplitPartials* acc, int row0, cudaStream_t st);
cudaError_t launch_qkv_finish(const SplitPartials& sp, const void* bias, const int* pos, const float2* rope, void* q,
                              void* k, void* v, int M, int Hq, int Hkv, cudaStream_t st);
cudaError_t launch_attn_tc(const AttnParams& a, int units_bound, bool clustered, cudaStream_t st);
cudaError_t launch_attn_f32(const AttnParams& a, int n_rows, cudaStream_t st);
cudaError_t launch_wait_probe(int* err, unsigned long long* waited_ns, unsigned long long limit_ns, cudaStream_t st);
cudaError_t gemm_prepare();
cudaError_t attn_prepare(int* max_clusters);
}  // namespace jf

using namespace jf;

namespace {

constexpr int kTargetCTAs = 152;   // split-K target: about one CTA per SM of a GB300
constexpr int kMaxGemmGrid = 256;  // persistent GEMM grids (one CTA per SM) never exceed this
// kernel classes of jf_kernel_time (include/jf.h)
enum ProfClass : int {
  PC_GATEUP = 0, PC_ATTN = 1, PC_GEMMS = 2, PC_QKV = 3, PC_OPROJ = 4, PC_DOWN = 5, PC_LMHEAD = 6, PC_RESERVED = 7,
  PC_NORM = 8, PC_OTHER = 9, kProfClasses = 10
};
constexpr int kMaxStateInts = 32768;

size_t rup(size_t x, size_t a) { return (x + a - 1) / a * a; }
int cdiv(long long a, long long b) { return (int)((a + b - 1) / b); }

int splits_for(int n_tiles, int kb_total) {
  if (n_tiles >= kTargetCTAs / 2) return 1;
  int s = kTargetCTAs / n_tiles;
  int cap = std::max(1, kb_total / 4);
  return std::max(1, std::min(std::min(s, cap), 8));   // the kernel reduces at most 8 splits
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

bool get_encode() {
  if (g_encode) return true;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !fn)
    return false;
  g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  return true;
}

// bf16 matrix [rows][K] (K contiguous) as a TMA tensor: boxes of 64 x box_rows, 128-byte swizzle.
bool make_tmap(CUtensorMap* tm, const void* ptr, long long K, long long rows, int box_rows) {
  if (!get_encode()) return false;
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  cuuint32_t box[2] = {(cuuint32_t)kTileK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// ------------------------------------------------------------------------------------------
// Arena plan: offsets of every device buffer, shared by jf_arena_bytes and jf_create.
// ------------------------------------------------------------------------------------------
struct Dims {
  int L, d, Hq, Hkv, hd, F, V, nq, nkv, nqkv, G;
  int es;
  bool bf16;
  bool qkv_bias, tie;  // per-feature Q/K/V biases; LM head = embedding matrix
  int R, S, max_ctx, pps, n_pages, logits_rows;
  int max_chains, max_units;
  int n_vtiles;
};

struct Plan {
  size_t total = 0;
  size_t take(size_t bytes, size_t align = 256) {
    total = rup(total, align);
    size_t o = total;
    total += bytes;
    return o;
  }
};

struct Offsets {
  size_t w_embed, w_lm, g_final, rope;
  std::vector<size_t> w_qkv, w_o, w_gu, w_d, g_attn, g_mlp, b_qkv;
  size_t k_pages, v_pages, page_table, seq_len, commit;
  size_t k_inf, v_inf, x, h, q, att, act;
  size_t tok, pos, gpred, top2, chains, n_chains, attn_xchg, attn_ticket;
  size_t gemm_ws, gemm_counter, am_v1, am_i1, am_v2, am_counter;
  size_t logits, err, traj_count;
  size_t gen_state, gen_out, gen_truth, gen_log, gen_q0, gen_plast, gen_prompt, gen_seqp, res, step_blocks, step_res,
      committed;
  size_t gemm_ws_bytes;
  size_t total;
};

jf_status make_dims(const jf_model_config* m, const jf_runtime_config* rt, Dims* D, std::string* why) {
  if (!m || !rt) { *why = "null config"; return JF_EINVAL; }
  if (m->n_layers < 1 || m->d_model < 64 || m->n_heads < 1 || m->n_kv_heads < 1 || m->head_dim < 2 || m->d_ff < 64 ||
      m->vocab < 2 || !(m->rms_eps >= 0) || !(m->rope_theta > 0)) {
    *why = "model dimensions out of range";
    return JF_EINVAL;
  }
  if (m->dtype != JF_F32 && m->dtype != JF_BF16) { *why = "dtype must be JF_F32 or JF_BF16"; return JF_EINVAL; }
  if ((m->qkv_bias != 0 && m->qkv_bias != 1) || (m->tie_embeddings != 0 && m->tie_embeddings != 1)) {
    *why = "qkv_bias and tie_embeddings must be 0 or 1";
    return JF_EINVAL;
  }
  if (m->n_heads % m->n_kv_heads) { *why = "n_heads must be a multiple of n_kv_heads"; return JF_EUNSUPPORTED; }
  if (m->dtype == JF_BF16 && m->head_dim != 128) { *why = "bf16 kernels need head_dim 128"; return JF_EUNSUPPORTED; }
  if (m->dtype == JF_F32 && m->head_dim != 64 && m->head_dim != 128) { *why = "head_dim must be 64 or 128"; return JF_EUNSUPPORTED; }
  if ((m->n_heads * m->head_dim) % 128 || (m->n_kv_heads * m->head_dim) % 128) {
    *why = "n_heads*head_dim and n_kv_heads*head_dim must be multiples of 128";
    return JF_EUNSUPPORTED;
  }
  if (m->d_model % 64 || m->d_ff % 64) { *why = "d_model and d_ff must be multiples of 64"; return JF_EUNSUPPORTED; }
  if (m->d_model > 8192) { *why = "d_model above 8192 is not supported by the norm kernel"; return JF_EUNSUPPORTED; }
  if (rt->max_seqs < 1 || rt->max_seqs > kMaxSeqs || rt->max_ctx < 16 || rt->max_rows < 1 || rt->max_rows > 4096 ||
      rt->logits_rows < 0 || rt->logits_rows > rt->max_rows) {
    *why = "runtime capacity out of range (max_seqs 1..64, max_ctx >= 16, max_rows 1..4096, logits_rows <= max_rows)";
    return JF_EINVAL;
  }
  if (m->dtype == JF_BF16 && rt->max_ctx > kAttnMaxCtx - kAttnChunk) {
    *why = "max_ctx above the bf16 attention's page-id staging capacity (130944 positions)";
    return JF_EINVAL;
  }
  D->L = m->n_layers; D->d = m->d_model; D->Hq = m->n_heads; D->Hkv = m->n_kv_heads; D->hd = m->head_dim;
  D->F = m->d_ff; D->V = m->vocab;
  D->nq = D->Hq * D->hd; D->nkv = D->Hkv * D->hd; D->nqkv = D->nq + 2 * D->nkv; D->G = D->Hq / D->Hkv;
  D->bf16 = m->dtype == JF_BF16; D->es = D->bf16 ? 2 : 4;
  D->qkv_bias = m->qkv_bias != 0; D->tie = m->tie_embeddings != 0;
  D->R = rt->max_rows; D->S = rt->max_seqs; D->max_ctx = rt->max_ctx;
  D->pps = cdiv(rt->max_ctx, kPage); D->n_pages = D->S * D->pps; D->logits_rows = rt->logits_rows;
  if (rt->page_size != 0 && rt->page_size != kPage) {
    *why = "page_size must be 16 (or 0 for the default)";
    return JF_EUNSUPPORTED;
  }
  if (rt->max_segments < 0 || rt->max_segments > kMaxChains) {
    *why = "max_segments out of range (0 = default, at most 256)";
    return JF_EINVAL;
  }
  D->max_chains = rt->max_segments > 0 ? rt->max_segments : std::min(kMaxChains, D->S * 5 + 1);
  if (D->bf16) {
    D->max_units = D->Hkv * (cdiv((long long)D->R * D->G, kAttnQRows) + D->max_chains);
  } else {
    D->max_units = 1;
  }
  D->n_vtiles = cdiv(D->V, kTileN);
  return JF_OK;
}

size_t gemm_ws_floats(const Dims& D) {
  if (!D.bf16) return 0;
  const int N[5] = {D.nqkv, D.d, 2 * D.F, D.d, D.V};
  const int K[5] = {D.d, D.nq, D.d, D.F, D.d};
  size_t mx = 0;
  for (int i = 0; i < 5; ++i) {
    const int nt = cdiv(N[i], kTileN), kb = cdiv(K[i], kTileK);
    const int sp = splits_for(nt, kb);
    // QKV, O and down always leave partial tiles for their consumer; the others only when split
    if (sp <= 1 && (i == 2 || i == 4)) continue;
    mx = std::max(mx, (size_t)sp * nt * ((size_t)D.R + 256) * kTileN);
  }
  return mx;
}

Offsets plan_offsets(const Dims& D) {
  Offsets o;
  Plan p;
  const size_t es = D.es;
  o.w_embed = p.take((size_t)D.V * D.d * es, 1024);
  o.w_lm = D.tie ? o.w_embed : p.take((size_t)D.V * D.d * es, 1024);
  o.g_final = p.take((size_t)D.d * 4);
  for (int l = 0; l < D.L; ++l) {
    o.w_qkv.push_back(p.take((size_t)D.nqkv * D.d * es, 1024));
    o.w_o.push_back(p.take((size_t)D.d * D.nq * es, 1024));
    o.w_gu.push_back(p.take((size_t)2 * D.F * D.d * es, 1024));
    o.w_d.push_back(p.take((size_t)D.d * D.F * es, 1024));
    o.g_attn.push_back(p.take((size_t)D.d * 4));
    o.g_mlp.push_back(p.take((size_t)D.d * 4));
    o.b_qkv.push_back(D.qkv_bias ? p.take((size_t)D.nqkv * es) : 0);  // model dtype, q | k | v
  }
  o.rope = p.take((size_t)(D.max_ctx + 1) * (D.hd / 2) * sizeof(float2));
  const size_t kv_layer = (size_t)D.n_pages * D.Hkv * kPage * D.hd * es;
  o.k_pages = p.take(kv_layer * D.L, 1024);
  o.v_pages = p.take(kv_layer * D.L, 1024);
  o.page_table = p.take((size_t)D.S * D.pps * 4);
  o.seq_len = p.take((size_t)D.S * 4);
  o.commit = p.take((size_t)D.S * sizeof(CommitInfo));
  const size_t inf_layer = (size_t)D.R * D.nkv * es;
  o.k_inf = p.take(inf_layer * D.L, 1024);
  o.v_inf = p.take(inf_layer * D.L, 1024);
  o.x = p.take((size_t)D.R * D.d * 4, 1024);
  o.h = p.take((size_t)D.R * D.d * es, 1024);
  o.q = p.take((size_t)D.R * D.nq * es, 1024);
  o.att = p.take((size_t)D.R * D.nq * es, 1024);
  o.act = p.take((size_t)D.R * D.F * es, 1024);
  o.tok = p.take((size_t)D.R * 4);
  o.pos = p.take((size_t)D.R * 4);
  o.gpred = p.take((size_t)D.R * 4);
  o.top2 = p.take((size_t)D.R * 8);
  o.chains = p.take((size_t)kMaxChains * sizeof(Chain));
  o.n_chains = p.take(16);
  // attention lane states: [unit][lane][128 x 128 O, 128 m, 128 l] fp32 (bf16 path)
  o.attn_xchg = p.take(D.bf16 ? (size_t)D.max_units * kAttnLanes * kAttnXchgFloats * 4 : 16, 1024);
  o.attn_ticket = p.take((size_t)D.max_units * 4);
  o.gemm_ws_bytes = gemm_ws_floats(D) * 4;
  o.gemm_ws = p.take(std::max<size_t>(o.gemm_ws_bytes, 16), 1024);
  const int max_mt = cdiv(D.R, 16) + 1;
  o.gemm_counter = p.take((size_t)(D.n_vtiles + 8) * max_mt * 4 + (size_t)(cdiv(2 * D.F, kTileN) + 8) * max_mt * 4);
  o.am_v1 = p.take((size_t)D.R * std::max(D.n_vtiles, kMaxGemmGrid) * 4);  // [row][CTA slot]
  o.am_i1 = p.take((size_t)D.R * std::max(D.n_vtiles, kMaxGemmGrid) * 4);  // [row][CTA slot]
  o.am_v2 = p.take((size_t)D.R * std::max(D.n_vtiles, kMaxGemmGrid) * 4);  // [row][CTA slot]
  o.am_counter = p.take((size_t)max_mt * 4);
  o.logits = p.take((size_t)std::max(D.logits_rows, 1) * D.V * 4, 1024);
  o.err = p.take(16);
  o.traj_count = p.take(16);
  o.gen_state = p.take((size_t)D.S * kMaxStateInts * 4);
  o.gen_out = p.take((size_t)D.S * D.max_ctx * 4);
  o.gen_truth = p.take((size_t)D.S * D.max_ctx * 4);
  o.gen_log = p.take((size_t)D.max_ctx * D.S * 4);
  o.gen_q0 = p.take((size_t)D.S * 4);
  o.gen_plast = p.take((size_t)D.S * 4);
  o.gen_prompt = p.take((size_t)D.S * D.max_ctx * 4);
  o.gen_seqp = p.take((size_t)D.S * kSeqParams * 4);
  o.res = p.take(sizeof(IterResult));
  o.step_blocks = p.take(sizeof(StepBlocks));
  o.step_res = p.take(sizeof(StepResult));
  o.committed = p.take((size_t)D.R * 4);
  o.total = rup(p.total, 1024) + 1024;  // slack for base alignment
  return o;
}

struct LayerW {
  void *qkv, *o, *gu, *dn;
  void* b_qkv;  // [nq + 2 nkv] in the model dtype, or null
  float *g_attn, *g_mlp;
  CUtensorMap tm_qkv, tm_o, tm_gu, tm_dn;
};

struct GraphRec {
  cudaGraphExec_t exec = nullptr;
  long long kernels = 0;        // kernel nodes in the graph
  std::vector<cudaEvent_t> ev;  // profiling event pairs, in launch order
  std::vector<int> ev_class;
};

}  // namespace

// Shared with the allocation-free GEMM entry point (jf_noalloc.cu).
int jf::gemm_default_splits(int n_tiles, int kb_total) { return splits_for(n_tiles, kb_total); }
bool jf::encode_tmap_bf16(CUtensorMap* tm, const void* ptr, long long K, long long rows, int box_rows) {
  return make_tmap(tm, ptr, K, rows, box_rows);
}

struct jf_ctx {
  jf_model_config mc;
  jf_runtime_config rc;
  Dims D;
  Offsets O;
  char* base = nullptr;
  cudaStream_t st = nullptr;
  bool own_stream = false;
  int device = 0;
  int num_sms = 152;
  std::string last_error;
  bool weights_ready = false;
  // device pointers
  void *w_embed, *w_lm;
  float* g_final;
  std::vector<LayerW> layers;
  CUtensorMap tm_lm;
  float2* rope;
  void *k_pages, *v_pages;
  int *page_table, *seq_len;
  CommitInfo* commit;
  void *k_inf, *v_inf;
  float* x;
  void *h, *q, *att, *act;
  int *tok, *pos, *gpred;
  float* top2;
  Chain* chains;
  int* n_chains;
  float* attn_xchg;
  int* attn_ticket;
  int attn_max_clusters = 0;  // 8-CTA clusters of the attention resident at once
  int chains_bound = 1;  // most chains the next forward can have (sizes the attention launch)
  float* gemm_ws;
  int* gemm_counter;
  float *am_v1, *am_v2;
  int *am_i1, *am_counter;
  float* logits;
  int* err;
  int *gen_state, *gen_out, *gen_truth, *gen_log, *gen_q0, *gen_plast, *gen_prompt, *gen_seqp, *traj_count;
  IterResult* res_dev;
  StepBlocks* sb_dev;
  StepResult* sres_dev;
  int* committed_dev;
  // pinned host
  IterResult* res_host = nullptr;
  // host mirrors
  std::vector<int> h_seq_len;
  std::vector<std::vector<int>> h_pages;
  std::vector<int> free_pages;
  // graphs of the decode iteration, keyed by (state stride, rows)
  std::map<std::pair<int, int>, GraphRec> graphs;
  GenCfg graph_cfg;
  bool have_graph_cfg = false;
  // profiling
  bool profiling = false;
  double prof_ms[kProfClasses] = {};
  long long prof_n[kProfClasses] = {};
  std::vector<cudaEvent_t>* capture_events = nullptr;
  std::vector<int>* capture_classes = nullptr;
  long long launches = 0;  // libjf kernels launched (graph replays count their kernel nodes)
  unsigned long long wait_ns = kWaitLimitDefaultNs;  // limit of each bounded device wait
};

namespace {

jf_status fail(jf_ctx* c, jf_status s, const std::string& msg) {
  if (c) c->last_error = msg;
  return s;
}

#define CK(expr)                                                                                   \
  do {                                                                                             \
    cudaError_t e_ = (expr);                                                                       \
    if (e_ != cudaSuccess) return fail(c, JF_ECUDA, std::string(#expr) + ": " + cudaGetErrorString(e_)); \
  } while (0)

template <typename T>
T* at(jf_ctx* c, size_t off) {
  return reinterpret_cast<T*>(c->base + off);
}

jf_status check_err_word(jf_ctx* c, int code) {
  if (code == 0) return JF_OK;
  if (code == JF_DERR_TIMEOUT_TMA || code == JF_DERR_TIMEOUT_MMA || code == JF_DERR_TIMEOUT_EPI ||
      code == JF_DERR_TIMEOUT_PROBE)
    return fail(c, JF_ETIMEOUT, "device wait timed out (code " + std::to_string(code) + ")");
  return fail(c, JF_EDEVICE, "device bounds check failed (code " + std::to_string(code) + ")");
}

jf_status read_err(jf_ctx* c) {
  int e = 0;
  CK(cudaMemcpyAsync(&e, c->err, 4, cudaMemcpyDeviceToHost, c->st));
  CK(cudaStreamSynchronize(c->st));
  if (e) {
    int z = 0;
    cudaMemcpyAsync(c->err, &z, 4, cudaMemcpyHostToDevice, c->st);
    cudaStreamSynchronize(c->st);
  }
  return check_err_word(c, e);
}

// ------------------------------------------------------------------------------------------
// KV pages: a free list handing out 16-token pages; the order is scrambled so that a sequence's
// pages are not contiguous and every access goes through the page table.
// ------------------------------------------------------------------------------------------
void init_pages(jf_ctx* c) {
  const int n = c->D.n_pages;
  c->free_pages.resize(n);
  // multiplicative permutation of 0..n-1 (stride coprime to n), popped from the back
  int stride = 1;
  for (int s : {7919, 104729, 15485863, 3, 5}) {
    int a = s % n, b = n;
    while (b) { int t = a % b; a = b; b = t; }
    if (a == 1 && s % n != 0) { stride = s % n; break; }
  }
  for (int i = 0; i < n; ++i) c->free_pages[i] = (int)(((long long)i * stride) % n);
  c->h_pages.assign(c->D.S, {});
  c->h_seq_len.assign(c->D.S, 0);
}

jf_status ensure_pages(jf_ctx* c, int seq, int n_pos) {
  std::vector<int>& pg = c->h_pages[seq];
  const int need = cdiv(n_pos, kPage);
  if (need > c->D.pps) return fail(c, JF_ECAPACITY, "sequence longer than max_ctx");
  const int have = (int)pg.size();
  if (need <= have) return JF_OK;
  if ((int)c->free_pages.size() < need - have) return fail(c, JF_ECAPACITY, "KV pages exhausted");
  for (int i = have; i < need; ++i) {
    pg.push_back(c->free_pages.back());
    c->free_pages.pop_back();
  }
  CK(cudaMemcpyAsync(c->page_table + (size_t)seq * c->D.pps + have, pg.data() + have, (size_t)(need - have) * 4,
                     cudaMemcpyHostToDevice, c->st));
  return JF_OK;
}

jf_status release_pages(jf_ctx* c, int seq, int keep_pos) {
  std::vector<int>& pg = c->h_pages[seq];
  const int keep = cdiv(keep_pos, kPage);
  while ((int)pg.size() > keep) {
    c->free_pages.push_back(pg.back());
    pg.pop_back();
  }
  return JF_OK;
}

jf_status set_seq_len(jf_ctx* c, int seq, int len) {
  c->h_seq_len[seq] = len;
  CK(cudaMemcpyAsync(c->seq_len + seq, &c->h_seq_len[seq], 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaStreamSynchronize(c->st));
  return JF_OK;
}

// ------------------------------------------------------------------------------------------
// Forward pass launch sequence (one pass over M in-flight rows; Eq. 3).
// ------------------------------------------------------------------------------------------
// LM head of a forward: greedy argmax of every row, logits of every row, argmax of the last row
// only (prefill: only the token after the prompt is needed), or none (non-final prefill chunks).
enum LmMode { LM_ARGMAX = 0, LM_LOGITS = 1, LM_LAST = 2, LM_NONE = 3 };

void prof_begin(jf_ctx* c, int cls) {
  if (!c->capture_events) return;
  cudaEvent_t e;
  cudaEventCreate(&e);
  cudaEventRecordWithFlags(e, c->st, cudaEventRecordExternal);
  c->capture_events->push_back(e);
  c->capture_classes->push_back(cls);
}
void prof_end(jf_ctx* c) {
  if (!c->capture_events) return;
  cudaEvent_t e;
  cudaEventCreate(&e);
  cudaEventRecordWithFlags(e, c->st, cudaEventRecordExternal);
  c->capture_events->push_back(e);
  c->capture_classes->push_back(-1);
}

cudaError_t gemm(jf_ctx* c, const CUtensorMap& tmA, const void* W, const void* X, int N, int K, int M,
                 const GemmEpi& epi, int cls) {
  const Dims& D = c->D;
  GemmParams p;
  p.N = N; p.K = K; p.M = M;
  p.n_tiles = cdiv(N, kTileN);
  p.kb_total = cdiv(K, kTileK);
  p.ws = c->gemm_ws;
  p.tile_counter = c->gemm_counter;
  p.err = c->err;
  p.wait_ns = c->wait_ns;
  p.grid = c->num_sms;
  p.epi = epi;
  p.epi.M = M;
  p.epi.N = N;
  const bool pr = c->capture_events && cls >= 0;
  if (pr) prof_begin(c, cls);
  cudaError_t e;
  if (D.bf16) {
    const int bn = gemm_bn_for(M);
    p.m_tiles = cdiv(M, bn);
    p.k_splits = splits_for(p.n_tiles, p.kb_total);
    CUtensorMap tmB;
    if (!make_tmap(&tmB, X, K, M, bn)) return cudaErrorInvalidValue;
    e = launch_gemm_bf16(tmA, tmB, p, bn, c->st);
  } else {
    p.m_tiles = cdiv(M, 32);
    p.k_splits = 1;
    e = launch_gemm_f32(reinterpret_cast<const float*>(W), reinterpret_cast<const float*>(X), p, c->st);
  }
  if (pr) prof_end(c);
  return e;
}

cudaError_t enqueue_forward(jf_ctx* c, int M, LmMode lm) {
  const Dims& D = c->D;
  const float eps = (float)c->mc.rms_eps;
  cudaError_t e;
  prof_begin(c, PC_OTHER);
  e = launch_embed(c->w_embed, D.bf16, c->tok, c->x, M, D.d, D.V, c->err, c->st);
  prof_end(c);
  if (e != cudaSuccess) return e;
  const size_t inf_layer = (size_t)D.R * D.nkv * D.es;
  const size_t kv_layer = (size_t)D.n_pages * D.Hkv * kPage * D.hd * D.es;
  // bf16: the QKV, O and down projections leave split-K partial tiles; the QKV finish kernel and
  // the following RMSNorms add them (split order) instead of a last-CTA reduction in the GEMM
  const bool partials = D.bf16;
  const bool qkv_partial = partials && D.hd == kTileN;
  auto split_parts = [&](int N, int K) {
    const int bn = gemm_bn_for(M);
    return SplitPartials{c->gemm_ws, splits_for(cdiv(N, kTileN), cdiv(K, kTileK)), cdiv(M, bn), bn};
  };
  const SplitPartials sp_qkv = split_parts(D.nqkv, D.d), sp_o = split_parts(D.d, D.nq), sp_dn = split_parts(D.d, D.F);
  for (int l = 0; l < D.L; ++l) {
    LayerW& w = c->layers[l];
    char* kinf = reinterpret_cast<char*>(c->k_inf) + l * inf_layer;
    char* vinf = reinterpret_cast<char*>(c->v_inf) + l * inf_layer;
    prof_begin(c, PC_NORM);
    e = launch_rmsnorm(c->x, w.g_attn, c->h, D.bf16, M, D.d, eps, (partials && l > 0) ? &sp_dn : nullptr, 0, c->st);
    prof_end(c);
    if (e != cudaSuccess) return e;
    GemmEpi ep = {};
    ep.kind = qkv_partial ? EPI_PARTIAL : EPI_QKV;
    ep.q_out = c->q; ep.k_out = kinf; ep.v_out = vinf;
    ep.n_q = D.nq; ep.n_kv = D.nkv; ep.head_dim = D.hd;
    ep.pos = c->pos; ep.rope = c->rope;
    ep.bias = w.b_qkv;
    if ((e = gemm(c, w.tm_qkv, w.qkv, c->h, D.nqkv, D.d, M, ep, PC_QKV)) != cudaSuccess) return e;
    if (qkv_partial) {
      prof_begin(c, PC_QKV);
      e = launch_qkv_finish(sp_qkv, w.b_qkv, c->pos, c->rope, c->q, kinf, vinf, M, D.Hq, D.Hkv, c->st);
      prof_end(c);
      if (e != cudaSuccess) return e;
    }
    AttnParams a = {};
    a.q = c->q; a.k_inf = kinf; a.v_inf = vinf;
    a.k_pages = reinterpret_cast<char*>(c->k_pages) + l * kv_layer;
    a.v_pages = reinterpret_cast<char*>(c->v_pages) + l * kv_layer;
    a.page_table = c->page_table; a.pages_per_seq = D.pps; a.n_pages = D.n_pages;
    a.seq_len = c->seq_len; a.chains = c->chains; a.n_chains_dev = c->n_chains;
    a.out = c->att; a.Hq = D.Hq; a.Hkv = D.Hkv; a.hd = D.hd;
    a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D.hd));
    a.err = c->err;
    a.wait_ns = c->wait_ns;
    a.xchg = c->attn_xchg;
    a.unit_ticket = c->attn_ticket;
    prof_begin(c, PC_ATTN);
    if (D.bf16) {
      // units of this forward are bounded by its rows: every chain adds at most one partial tile
      const int units_bound = std::min(D.max_units, D.Hkv * (cdiv((long long)M * D.G, kAttnQRows) + c->chains_bound));
      // clustered unless the unclustered form needs fewer waves of units (jf_attn_form.h)
      const int units_est = attn_units_estimate(M, c->chains_bound, units_bound, D.Hkv, D.G, kAttnQRows);
      e = launch_attn_tc(a, units_bound, attn_use_clusters(units_est, kAttnLanes, c->attn_max_clusters, c->num_sms),
                         c->st);
      prof_end(c);
    } else {
      e = launch_attn_f32(a, M, c->st);
      prof_end(c);
    }
    if (e != cudaSuccess) return e;
    GemmEpi er = {};
    er.kind = partials ? EPI_PARTIAL : EPI_RESID; er.x = c->x; er.ldx = D.d;
    if ((e = gemm(c, w.tm_o, w.o, c->att, D.d, D.nq, M, er, PC_OPROJ)) != cudaSuccess) return e;
    prof_begin(c, PC_NORM);
    e = launch_rmsnorm(c->x, w.g_mlp, c->h, D.bf16, M, D.d, eps, partials ? &sp_o : nullptr, 0, c->st);
    prof_end(c);
    if (e != cudaSuccess) return e;
    GemmEpi es = {};
    es.kind = EPI_SWIGLU; es.act = c->act; es.ld_act = D.F;
    if ((e = gemm(c, w.tm_gu, w.gu, c->h, 2 * D.F, D.d, M, es, PC_GATEUP)) != cudaSuccess) return e;
    if ((e = gemm(c, w.tm_dn, w.dn, c->act, D.d, D.F, M, er, PC_DOWN)) != cudaSuccess) return e;
  }
  if (lm == LM_NONE) {
    c->launches += 1 + (qkv_partial ? 8LL : 7LL) * D.L;
    return cudaSuccess;
  }
  const int lm_rows = (lm == LM_LAST) ? 1 : M;
  prof_begin(c, PC_NORM);
  e = launch_rmsnorm(c->x, c->g_final, c->h, D.bf16, lm_rows, D.d, eps, (partials && D.L > 0) ? &sp_dn : nullptr,
                     M - lm_rows, c->st);
  prof_end(c);
  if (e != cudaSuccess) return e;
  GemmEpi el = {};
  if (lm != LM_LOGITS) {
    el.kind = EPI_ARGMAX;
    el.am_v1 = c->am_v1; el.am_i1 = c->am_i1; el.am_v2 = c->am_v2; el.am_counter = c->am_counter;
    el.am_out = c->gpred; el.top2_out = c->top2;
  } else {
    el.kind = EPI_STORE; el.y = c->logits; el.ldy = D.V;
  }
  c->launches += 1 + (qkv_partial ? 8LL : 7LL) * D.L + 2;
  return gemm(c, c->tm_lm, c->w_lm, c->h, D.V, D.d, lm_rows, el, PC_LMHEAD);
}

// Upload the rows of one causal chain of sequence `seq` (positions P .. P+M-1).
jf_status upload_chain(jf_ctx* c, int seq, int P, int M, const int32_t* tokens_host, const int32_t* tokens_dev) {
  std::vector<int> pos(M);
  for (int i = 0; i < M; ++i) pos[i] = P + i;
  Chain ch{seq, 0, M, P};
  int one = 1;
  if (tokens_dev) CK(cudaMemcpyAsync(c->tok, tokens_dev, (size_t)M * 4, cudaMemcpyDeviceToDevice, c->st));
  else CK(cudaMemcpyAsync(c->tok, tokens_host, (size_t)M * 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->pos, pos.data(), (size_t)M * 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->chains, &ch, sizeof(Chain), cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->n_chains, &one, 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaStreamSynchronize(c->st));
  c->chains_bound = 1;
  return JF_OK;
}

jf_status check_tokens(jf_ctx* c, const int32_t* t, int n) {
  for (int i = 0; i < n; ++i)
    if (t[i] < 0 || t[i] >= c->D.V) return fail(c, JF_EINVAL, "token id out of range");
  return JF_OK;
}

// Prefill of `len` tokens (host or device) of sequence `seq`; q0 -> *next (host).
jf_status prefill_impl(jf_ctx* c, int seq, const int32_t* host_prompt, const int32_t* dev_prompt, int len,
                       int32_t* next) {
  const Dims& D = c->D;
  const int P0 = c->h_seq_len[seq];
  jf_status s;
  if ((s = ensure_pages(c, seq, P0 + len)) != JF_OK) return s;
  int P = P0;
  for (int start = 0; start < len; start += D.R) {
    const int m = std::min(D.R, len - start);
    s = upload_chain(c, seq, P, m, host_prompt ? host_prompt + start : nullptr, dev_prompt ? dev_prompt + start : nullptr);
    if (s != JF_OK) return s;
    const bool last_chunk = start + m >= len;
    CK(enqueue_forward(c, m, last_chunk ? LM_LAST : LM_NONE));
    CommitInfo ci{0, m, P};
    CK(cudaMemcpyAsync(c->commit + seq, &ci, sizeof(ci), cudaMemcpyHostToDevice, c->st));
    CK(launch_commit(c->commit + seq, 1, D.L, c->k_inf, c->v_inf, c->k_pages, c->v_pages,
                     c->page_table + (size_t)seq * D.pps, D.pps, D.n_pages, D.R, D.Hkv, D.hd, D.es, c->seq_len + seq,
                     c->err, c->st));
    c->launches += 1;
    P += m;
    if (start + m >= len) {
      int32_t q0 = -1;
      CK(cudaMemcpyAsync(&q0, c->gpred, 4, cudaMemcpyDeviceToHost, c->st));
      CK(cudaStreamSynchronize(c->st));
      if (next) *next = q0;
    }
  }
  if ((s = read_err(c)) != JF_OK) return s;
  c->h_seq_len[seq] = P;
  return JF_OK;
}

// ------------------------------------------------------------------------------------------
// Decode iteration graph: forward(M) + acceptance/state update + KV commit + result readback.
// ------------------------------------------------------------------------------------------
cudaError_t enqueue_iteration(jf_ctx* c, const GenCfg& g, int M, int n_seqs) {
  const Dims& D = c->D;
  cudaError_t e = enqueue_forward(c, M, LM_ARGMAX);
  if (e != cudaSuccess) return e;
  prof_begin(c, PC_OTHER);
  e = launch_gen_accept(g, c->gen_state, c->gpred, M, c->tok, c->pos, c->chains, c->n_chains, c->commit, c->res_dev,
                        c->err, c->st);
  prof_end(c);
  if (e != cudaSuccess) return e;
  prof_begin(c, PC_OTHER);
  e = launch_commit(c->commit, n_seqs, D.L, c->k_inf, c->v_inf, c->k_pages, c->v_pages, c->page_table, D.pps,
                    D.n_pages, D.R, D.Hkv, D.hd, D.es, c->seq_len, c->err, c->st);
  prof_end(c);
  if (e != cudaSuccess) return e;
  c->launches += 2;
  return cudaMemcpyAsync(c->res_host, c->res_dev, sizeof(IterResult), cudaMemcpyDeviceToHost, c->st);
}

bool same_cfg(const GenCfg& a, const GenCfg& b) { return std::memcmp(&a, &b, sizeof(GenCfg)) == 0; }

void drop_graphs(jf_ctx* c) {
  for (auto& kv : c->graphs) {
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
    for (cudaEvent_t e : kv.second.ev) cudaEventDestroy(e);
  }
  c->graphs.clear();
}

jf_status get_graph(jf_ctx* c, const GenCfg& g, int M, int n_seqs, GraphRec** out) {
  if (!c->have_graph_cfg || !same_cfg(c->graph_cfg, g)) {
    drop_graphs(c);
    c->graph_cfg = g;
    c->have_graph_cfg = true;
  }
  const auto key = std::make_pair(c->profiling ? 1 : 0, M);
  auto it = c->graphs.find(key);
  if (it != c->graphs.end()) {
    *out = &it->second;
    return JF_OK;
  }
  GraphRec rec;
  CK(cudaStreamBeginCapture(c->st, cudaStreamCaptureModeThreadLocal));
  if (c->profiling) {
    c->capture_events = &rec.ev;
    c->capture_classes = &rec.ev_class;
  }
  const long long before = c->launches;
  cudaError_t e = enqueue_iteration(c, g, M, n_seqs);
  rec.kernels = c->launches - before;
  c->launches = before;
  c->capture_events = nullptr;
  c->capture_classes = nullptr;
  cudaGraph_t graph = nullptr;
  cudaError_t e2 = cudaStreamEndCapture(c->st, &graph);
  if (e != cudaSuccess || e2 != cudaSuccess) {
    if (graph) cudaGraphDestroy(graph);
    for (cudaEvent_t ev : rec.ev) cudaEventDestroy(ev);
    return fail(c, JF_ECUDA, std::string("graph capture failed: ") + cudaGetErrorString(e != cudaSuccess ? e : e2));
  }
  e = cudaGraphInstantiate(&rec.exec, graph, 0);
  cudaGraphDestroy(graph);
  if (e != cudaSuccess) {
    for (cudaEvent_t ev : rec.ev) cudaEventDestroy(ev);
    return fail(c, JF_ECUDA, std::string("graph instantiate: ") + cudaGetErrorString(e));
  }
  auto ins = c->graphs.emplace(key, rec);
  *out = &ins.first->second;
  return JF_OK;
}

void accumulate_profile(jf_ctx* c, GraphRec* g) {
  for (size_t i = 0; i + 1 < g->ev.size(); ++i) {
    const int cls = g->ev_class[i];
    if (cls < 0) continue;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, g->ev[i], g->ev[i + 1]) == cudaSuccess) {
      c->prof_ms[cls] += ms;
      c->prof_n[cls] += 1;
      if (cls == PC_GATEUP || cls == PC_QKV || cls == PC_OPROJ || cls == PC_DOWN || cls == PC_LMHEAD) {
        c->prof_ms[PC_GEMMS] += ms;
        c->prof_n[PC_GEMMS] += 1;
      }
    }
  }
}

// Timing events of one call; destroyed on every return path (an event still pending in the stream
// is released once the device reaches it).
struct CallEvents {
  cudaEvent_t e[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
  ~CallEvents() {
    for (cudaEvent_t x : e)
      if (x) cudaEventDestroy(x);
  }
};

jf_status generate_impl(jf_ctx* c, int n_seqs, const int32_t* const* h_prompts, const int32_t* d_prompts,
                        const int32_t* prompt_lens, const jf_gen_params* gp, int32_t* h_out, int32_t* d_out,
                        jf_gen_stats* stats, bool device_io) {
  const Dims& D = c->D;
  if (!c->weights_ready) return fail(c, JF_ESTATE, "weights not initialised");
  if (!gp || n_seqs < 1 || n_seqs > D.S || !prompt_lens) return fail(c, JF_EINVAL, "bad n_seqs / params");
  jf_gen_params p = *gp;
  const bool ar = p.mode == JF_MODE_AR;
  if (ar) {
    p.mode = JF_MODE_WINDOW;
    p.block_size = 1;
    p.n_blocks = 1;
    p.pool_size = 0;
    p.cand_per_iter = 0;
  }
  if (p.mode != JF_MODE_BLOCK && p.mode != JF_MODE_WINDOW) return fail(c, JF_EINVAL, "mode");
  if (p.init != JF_INIT_REPEAT && p.init != JF_INIT_INJECT) return fail(c, JF_EINVAL, "init");
  if (p.block_size < 1 || p.n_blocks < 1 || p.n_blocks > 8 || p.max_new < 1 || p.pool_size < 0 || p.pool_size > 1024 ||
      p.cand_per_iter < 0 || p.cand_per_iter > 4 || p.ngram_len < 0 || !(p.spawn_ratio >= 0.0 && p.spawn_ratio <= 1.0))
    return fail(c, JF_EINVAL, "generation parameter out of range");
  if (p.n_blocks > 1 && p.mode != JF_MODE_BLOCK) return fail(c, JF_EINVAL, "multi-block decoding needs block mode");
  if (!(p.inject_p >= 0.f && p.inject_p <= 1.f)) return fail(c, JF_EINVAL, "inject_p must be in [0, 1]");
  const int G = p.ngram_len > 0 ? p.ngram_len : p.block_size;
  const int C = p.pool_size > 0 ? p.cand_per_iter : 0;
  const int rows_per_seq = p.n_blocks * p.block_size + C * G;  // at the largest block size
  if ((long long)n_seqs * (1 + C) > D.max_chains)
    return fail(c, JF_ECAPACITY, "more attention chains (sequences x (1 + candidates)) than max_segments");
  // per-sequence block sizes (serving several requests at once) and late joins (chunked prefill
  // inside the decode iterations)
  const int chunk = p.prefill_chunk > 0 ? p.prefill_chunk : std::min(64, D.R);
  std::vector<int> nb(n_seqs, p.block_size), join(n_seqs, 0);
  long long rows_total = 0;
  for (int b = 0; b < n_seqs; ++b) {
    if (p.block_sizes && !ar) nb[b] = p.block_sizes[b];
    if (p.join_iters) join[b] = p.join_iters[b];
    if (nb[b] < 1 || nb[b] > p.block_size) return fail(c, JF_EINVAL, "block_sizes[b] must be in 1..block_size");
    if (join[b] < 0 || join[b] > (1 << 20)) return fail(c, JF_EINVAL, "join_iters[b] out of range");
    const int rb = p.n_blocks * nb[b] + C * std::min(G, nb[b]);  // candidates are cut to the draft length
    rows_total += join[b] > 0 ? std::max(rb, chunk) : rb;
  }
  if (chunk > D.R && std::any_of(join.begin(), join.end(), [](int j) { return j > 0; }))
    return fail(c, JF_EINVAL, "prefill_chunk exceeds max_rows");
  if (rows_total > D.R) return fail(c, JF_ECAPACITY, "in-flight rows exceed max_rows");
  if (1 + C > 5) return fail(c, JF_EINVAL, "too many candidates");
  const SeqLayout L = seq_layout(p.block_size, p.n_blocks, C, G, p.pool_size);
  if (L.total > kMaxStateInts || (size_t)(L.total + D.R) * 4 > 200 * 1024)
    return fail(c, JF_ECAPACITY, "decoding state too large (block size x blocks, pool x n-gram)");
  const int need_truth = p.max_new + p.n_blocks * p.block_size + G + 1;
  if (p.init == JF_INIT_INJECT && (!p.truth || p.truth_len < need_truth || p.truth_len > D.max_ctx))
    return fail(c, JF_EINVAL, "inject mode needs truth with truth_len >= max_new + K*n + G + 1 (and <= max_ctx)");
  std::vector<int> plen(n_seqs);
  long long poff_total = 0;
  for (int b = 0; b < n_seqs; ++b) {
    plen[b] = prompt_lens[b];
    if (plen[b] < 1) return fail(c, JF_EINVAL, "empty prompt");
    if (plen[b] + p.max_new + rows_per_seq + 2 > D.max_ctx) return fail(c, JF_ECAPACITY, "prompt + max_new exceeds max_ctx");
    if (!device_io) {
      if (!h_prompts || !h_prompts[b]) return fail(c, JF_EINVAL, "null prompt");
      jf_status s = check_tokens(c, h_prompts[b], plen[b]);
      if (s != JF_OK) return s;
    }
    poff_total += plen[b];
  }
  if (!device_io && p.init == JF_INIT_INJECT) {
    jf_status s = check_tokens(c, p.truth, n_seqs * p.truth_len);
    if (s != JF_OK) return s;
  }
  const bool want_traj = stats && stats->traj;
  if (want_traj && (stats->traj_cap < 1 || stats->traj_rows < rows_total))
    return fail(c, JF_EINVAL, "trajectory buffer: traj_cap >= 1 and traj_rows >= the rows of one forward needed");
  // reset slots 0 .. n_seqs-1 and reserve their pages
  for (int b = 0; b < n_seqs; ++b) {
    release_pages(c, b, 0);
    c->h_seq_len[b] = 0;
  }
  std::vector<int> zeros(n_seqs, 0);
  CK(cudaMemcpyAsync(c->seq_len, zeros.data(), (size_t)n_seqs * 4, cudaMemcpyHostToDevice, c->st));
  for (int b = 0; b < n_seqs; ++b) {
    jf_status s = ensure_pages(c, b, plen[b] + p.max_new + rows_per_seq + 2);
    if (s != JF_OK) return s;
  }
  const long long launches0 = c->launches;
  CallEvents ev;  // released on every return path
  CK(cudaEventCreate(&ev.e[0]));
  CK(cudaEventCreate(&ev.e[1]));
  CK(cudaEventCreate(&ev.e[2]));
  const cudaEvent_t e0 = ev.e[0], e1 = ev.e[1], e2 = ev.e[2];
  const bool time_iters = stats && stats->iter_ms && stats->accepted_cap > 0;
  if (time_iters) {  // around each graph replay, outside the graph
    CK(cudaEventCreate(&ev.e[3]));
    CK(cudaEventCreate(&ev.e[4]));
  }
  CK(cudaEventRecord(e0, c->st));
  std::vector<int> q0(n_seqs, 0), plast(n_seqs, 0), seqp((size_t)n_seqs * kSeqParams, 0);
  long long off = 0, loff = 0;  // offsets in the caller's prompts and in the late prompts' buffer
  for (int b = 0; b < n_seqs; ++b) {
    int* sp = &seqp[(size_t)b * kSeqParams];
    sp[SP_N] = nb[b];
    sp[SP_SSPAWN] = (int)std::ceil(p.spawn_ratio * nb[b] - 1e-12);
    sp[SP_JOIN] = join[b];
    sp[SP_PLEN] = plen[b];
    if (join[b] > 0) {
      // prefilled later, inside the decode iterations: keep its prompt on the device
      if (loff + plen[b] > (long long)D.S * D.max_ctx) return fail(c, JF_ECAPACITY, "late prompts exceed their buffer");
      sp[SP_POFF] = (int)loff;
      CK(cudaMemcpyAsync(c->gen_prompt + loff, device_io ? d_prompts + off : h_prompts[b], (size_t)plen[b] * 4,
                         device_io ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, c->st));
      loff += plen[b];
    } else {
      int32_t nt = -1;
      jf_status s = prefill_impl(c, b, device_io ? nullptr : h_prompts[b], device_io ? d_prompts + off : nullptr, plen[b], &nt);
      if (s != JF_OK) return s;
      q0[b] = nt;
      if (device_io) CK(cudaMemcpy(&plast[b], d_prompts + off + plen[b] - 1, 4, cudaMemcpyDeviceToHost));
      else plast[b] = h_prompts[b][plen[b] - 1];
    }
    off += plen[b];
  }
  CK(cudaMemcpyAsync(c->gen_seqp, seqp.data(), seqp.size() * 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaEventRecord(e1, c->st));
  CK(cudaMemcpyAsync(c->gen_q0, q0.data(), (size_t)n_seqs * 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->gen_plast, plast.data(), (size_t)n_seqs * 4, cudaMemcpyHostToDevice, c->st));
  if (p.init == JF_INIT_INJECT) {
    CK(cudaMemcpyAsync(c->gen_truth, p.truth, (size_t)n_seqs * p.truth_len * 4,
                       device_io ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, c->st));
  }
  CK(cudaMemsetAsync(c->gen_log, 0xff, (size_t)D.max_ctx * n_seqs * 4, c->st));
  CK(cudaMemsetAsync(c->gen_out, 0xff, (size_t)n_seqs * p.max_new * 4, c->st));
  GenCfg g = {};
  g.n = p.block_size; g.K = p.n_blocks;
  g.s_spawn = (int)std::ceil(p.spawn_ratio * p.block_size - 1e-12);
  g.pool_size = p.pool_size; g.G = G; g.C = C;
  g.mode = p.mode == JF_MODE_WINDOW ? GM_WINDOW : GM_BLOCK;
  g.init = p.init == JF_INIT_INJECT ? GI_INJECT : GI_REPEAT;
  g.T = (unsigned long long)((double)p.inject_p * 9007199254740992.0);
  g.seed = p.seed;
  g.max_new = p.max_new; g.eos = p.eos_id; g.V = D.V; g.n_seqs = n_seqs;
  g.truth = c->gen_truth; g.truth_stride = p.init == JF_INIT_INJECT ? p.truth_len : 0;
  g.truth_len = p.init == JF_INIT_INJECT ? p.truth_len : 0;
  g.state_stride = L.total;
  g.max_rows = D.R; g.max_chains = D.max_chains; g.max_ctx = D.max_ctx;
  c->chains_bound = std::min(D.max_chains, n_seqs * (1 + g.C));  // a prefilling sequence has one chain
  g.out_tokens = c->gen_out; g.iter_log = c->gen_log; g.max_iters = D.max_ctx;
  g.seq_params = c->gen_seqp;
  g.prompts = c->gen_prompt;
  g.prefill_chunk = chunk;
  if (want_traj) {
    g.traj = stats->traj;
    g.traj_cap = stats->traj_cap;
    g.traj_rows = stats->traj_rows;
    g.traj_count = c->traj_count;
    CK(cudaMemsetAsync(c->traj_count, 0, 4, c->st));
  }
  CK(launch_gen_init(g, c->gen_state, c->gen_q0, c->seq_len, c->gen_plast, c->tok, c->pos, c->chains, c->n_chains,
                     c->res_dev, c->err, c->st));
  c->launches += 1;
  CK(cudaMemcpyAsync(c->res_host, c->res_dev, sizeof(IterResult), cudaMemcpyDeviceToHost, c->st));
  CK(cudaStreamSynchronize(c->st));
  jf_status s = check_err_word(c, c->res_host->err);
  if (s != JF_OK) return s;
  int M = c->res_host->next_M;
  int iters = 0;
  std::vector<int> rows_log;
  bool done = c->res_host->all_done != 0;
  while (!done) {
    if (M < 1 || M > D.R) return fail(c, JF_EDEVICE, "device produced an invalid row count");
    GraphRec* gr = nullptr;
    if ((s = get_graph(c, g, M, n_seqs, &gr)) != JF_OK) return s;
    if (time_iters) CK(cudaEventRecord(ev.e[3], c->st));
    CK(cudaGraphLaunch(gr->exec, c->st));
    if (time_iters) CK(cudaEventRecord(ev.e[4], c->st));
    c->launches += gr->kernels;
    CK(cudaStreamSynchronize(c->st));
    if (time_iters && iters < stats->accepted_cap) {
      float ms = 0.f;
      CK(cudaEventElapsedTime(&ms, ev.e[3], ev.e[4]));
      stats->iter_ms[iters] = ms;
    }
    if (c->profiling) accumulate_profile(c, gr);
    rows_log.push_back(M);
    ++iters;
    if ((s = check_err_word(c, c->res_host->err)) != JF_OK) return s;
    done = c->res_host->all_done != 0;
    M = c->res_host->next_M;
    // every forward commits a token or a prefill chunk of some sequence
    if (iters > (long long)D.max_ctx * n_seqs + 16) return fail(c, JF_EDEVICE, "decoding did not terminate");
  }
  CK(cudaEventRecord(e2, c->st));
  if (device_io) {
    CK(cudaMemcpyAsync(d_out, c->gen_out, (size_t)n_seqs * p.max_new * 4, cudaMemcpyDeviceToDevice, c->st));
  } else {
    CK(cudaMemcpyAsync(h_out, c->gen_out, (size_t)n_seqs * p.max_new * 4, cudaMemcpyDeviceToHost, c->st));
  }
  CK(cudaStreamSynchronize(c->st));
  for (int b = 0; b < n_seqs; ++b) c->h_seq_len[b] = c->res_host->P[b];
  if (stats) {
    stats->iterations = iters;
    stats->kernel_launches = c->launches - launches0;
    stats->traj_iters = want_traj ? std::min(iters, stats->traj_cap) : 0;
    float a = 0.f, d2 = 0.f;
    cudaEventElapsedTime(&a, e0, e1);
    cudaEventElapsedTime(&d2, e1, e2);
    stats->prefill_ms = a;
    stats->decode_ms = d2;
    const int cap = std::min(stats->accepted_cap, iters);
    if (stats->accepted && cap > 0)
      CK(cudaMemcpy(stats->accepted, c->gen_log, (size_t)cap * n_seqs * 4, cudaMemcpyDeviceToHost));
    if (stats->rows)
      for (int i = 0; i < cap; ++i) stats->rows[i] = rows_log[i];
  }
  return JF_OK;
}

}  // namespace

// ==========================================================================================
// C ABI
// ==========================================================================================
extern "C" {

jf_status jf_arena_bytes(const jf_model_config* model, const jf_runtime_config* rt, size_t* out_bytes) {
  Dims D;
  std::string why;
  jf_status s = make_dims(model, rt, &D, &why);
  if (s != JF_OK) return s;
  if (!out_bytes) return JF_EINVAL;
  *out_bytes = plan_offsets(D).total;
  return JF_OK;
}

jf_status jf_create(const jf_model_config* model, const jf_runtime_config* rt, jf_ctx** out) {
  if (!out) return JF_EINVAL;
  *out = nullptr;
  Dims D;
  std::string why;
  jf_status s = make_dims(model, rt, &D, &why);
  if (s != JF_OK) return s;
  Offsets O = plan_offsets(D);
  if (!rt->device_arena || rt->arena_bytes < O.total) return JF_ENOMEM;
  jf_ctx* c = new jf_ctx();
  c->mc = *model;
  c->rc = *rt;
  c->D = D;
  c->O = O;
  c->base = reinterpret_cast<char*>(rup(reinterpret_cast<uintptr_t>(rt->device_arena), 1024));
  cudaGetDevice(&c->device);
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
  c->num_sms = std::min(c->num_sms, kMaxGemmGrid);
  if (rt->cuda_stream) {
    c->st = reinterpret_cast<cudaStream_t>(rt->cuda_stream);
  } else {
    if (cudaStreamCreateWithFlags(&c->st, cudaStreamNonBlocking) != cudaSuccess) { delete c; return JF_ECUDA; }
    c->own_stream = true;
  }
  // a failure from here on releases what the context already holds
  auto abandon = [c](jf_status s) {
    if (c->res_host) cudaFreeHost(c->res_host);
    if (c->own_stream) cudaStreamDestroy(c->st);
    delete c;
    return s;
  };
  c->w_embed = at<void>(c, O.w_embed);
  c->w_lm = at<void>(c, O.w_lm);
  c->g_final = at<float>(c, O.g_final);
  c->layers.resize(D.L);
  for (int l = 0; l < D.L; ++l) {
    LayerW& w = c->layers[l];
    w.qkv = at<void>(c, O.w_qkv[l]);
    w.o = at<void>(c, O.w_o[l]);
    w.gu = at<void>(c, O.w_gu[l]);
    w.dn = at<void>(c, O.w_d[l]);
    w.g_attn = at<float>(c, O.g_attn[l]);
    w.g_mlp = at<float>(c, O.g_mlp[l]);
    w.b_qkv = D.qkv_bias ? at<void>(c, O.b_qkv[l]) : nullptr;
    if (D.bf16) {
      bool ok = make_tmap(&w.tm_qkv, w.qkv, D.d, D.nqkv, kTileN) && make_tmap(&w.tm_o, w.o, D.nq, D.d, kTileN) &&
                make_tmap(&w.tm_gu, w.gu, D.d, 2 * D.F, kTileN) && make_tmap(&w.tm_dn, w.dn, D.F, D.d, kTileN);
      if (!ok) return abandon(JF_ECUDA);
    }
  }
  if (D.bf16 && !make_tmap(&c->tm_lm, c->w_lm, D.d, D.V, kTileN)) return abandon(JF_ECUDA);
  c->rope = at<float2>(c, O.rope);
  c->k_pages = at<void>(c, O.k_pages);
  c->v_pages = at<void>(c, O.v_pages);
  c->page_table = at<int>(c, O.page_table);
  c->seq_len = at<int>(c, O.seq_len);
  c->commit = at<CommitInfo>(c, O.commit);
  c->k_inf = at<void>(c, O.k_inf);
  c->v_inf = at<void>(c, O.v_inf);
  c->x = at<float>(c, O.x);
  c->h = at<void>(c, O.h);
  c->q = at<void>(c, O.q);
  c->att = at<void>(c, O.att);
  c->act = at<void>(c, O.act);
  c->tok = at<int>(c, O.tok);
  c->pos = at<int>(c, O.pos);
  c->gpred = at<int>(c, O.gpred);
  c->top2 = at<float>(c, O.top2);
  c->chains = at<Chain>(c, O.chains);
  c->attn_xchg = at<float>(c, O.attn_xchg);
  c->attn_ticket = at<int>(c, O.attn_ticket);
  c->n_chains = at<int>(c, O.n_chains);
  c->gemm_ws = at<float>(c, O.gemm_ws);
  c->gemm_counter = at<int>(c, O.gemm_counter);
  c->am_v1 = at<float>(c, O.am_v1);
  c->am_i1 = at<int>(c, O.am_i1);
  c->am_v2 = at<float>(c, O.am_v2);
  c->am_counter = at<int>(c, O.am_counter);
  c->logits = at<float>(c, O.logits);
  c->err = at<int>(c, O.err);
  c->gen_state = at<int>(c, O.gen_state);
  c->gen_out = at<int>(c, O.gen_out);
  c->gen_truth = at<int>(c, O.gen_truth);
  c->gen_log = at<int>(c, O.gen_log);
  c->gen_q0 = at<int>(c, O.gen_q0);
  c->gen_plast = at<int>(c, O.gen_plast);
  c->traj_count = at<int>(c, O.traj_count);
  c->gen_prompt = at<int>(c, O.gen_prompt);
  c->gen_seqp = at<int>(c, O.gen_seqp);
  c->res_dev = at<IterResult>(c, O.res);
  c->sb_dev = at<StepBlocks>(c, O.step_blocks);
  c->sres_dev = at<StepResult>(c, O.step_res);
  c->committed_dev = at<int>(c, O.committed);
  if (cudaMallocHost(&c->res_host, sizeof(IterResult)) != cudaSuccess) {
    c->res_host = nullptr;
    return abandon(JF_ENOMEM);
  }
  init_pages(c);
  // zero the small control buffers; fill the page table with -1
  cudaError_t e = cudaSuccess;
  auto zero = [&](size_t off, size_t bytes) {
    if (e == cudaSuccess) e = cudaMemsetAsync(c->base + off, 0, bytes, c->st);
  };
  zero(O.seq_len, (size_t)D.S * 4);
  zero(O.commit, (size_t)D.S * sizeof(CommitInfo));
  zero(O.gemm_counter, (O.am_v1 - O.gemm_counter));
  zero(O.am_counter, (size_t)(cdiv(D.R, 16) + 1) * 4);
  zero(O.err, 16);
  zero(O.attn_ticket, (size_t)D.max_units * 4);
  zero(O.n_chains, 16);
  zero(O.x, (size_t)D.R * D.d * 4);
  zero(O.h, (size_t)D.R * D.d * D.es);
  zero(O.act, (size_t)D.R * D.F * D.es);
  zero(O.att, (size_t)D.R * D.nq * D.es);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->page_table, 0xff, (size_t)D.S * D.pps * 4, c->st);
  if (e == cudaSuccess) e = launch_rope_table(c->rope, D.max_ctx + 1, D.hd / 2, c->mc.rope_theta, c->st);
  if (e == cudaSuccess) e = gemm_prepare();
  if (e == cudaSuccess) e = attn_prepare(&c->attn_max_clusters);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->st);
  if (e != cudaSuccess) return abandon(JF_ECUDA);
  *out = c;
  return JF_OK;
}

void jf_destroy(jf_ctx* c) {
  if (!c) return;
  if (c->st) cudaStreamSynchronize(c->st);
  drop_graphs(c);
  if (c->res_host) cudaFreeHost(c->res_host);
  if (c->own_stream) cudaStreamDestroy(c->st);
  delete c;
}

const char* jf_last_error(const jf_ctx* c) { return c ? c->last_error.c_str() : "null context"; }

}  // extern "C"

// ------------------------------------------------------------------------------------------
// Weights
// ------------------------------------------------------------------------------------------
namespace {

struct TensorLoc {
  char* base;        // device base of the (device-layout) tensor
  long long rows, cols;
  long long grp, grp_stride, grp_off;  // logical row r -> device row (r/grp)*grp_stride + r%grp + grp_off
  bool gain;         // fp32 RMSNorm gain (not a matrix)
};

bool tensor_loc(jf_ctx* c, int tid, TensorLoc* t) {
  const Dims& D = c->D;
  const long long big = 1ll << 40;
  *t = TensorLoc{nullptr, 0, 0, big, 0, 0, false};
  if (tid == 0) { t->base = (char*)c->w_embed; t->rows = D.V; t->cols = D.d; return true; }
  if (tid == 1) {
    if (D.tie) return false;  // tied: the embedding (tensor 0) is the LM head
    t->base = (char*)c->w_lm; t->rows = D.V; t->cols = D.d; return true;
  }
  if (tid == 2) { t->base = (char*)c->g_final; t->rows = 1; t->cols = D.d; t->gain = true; return true; }
  if (tid < 8) return false;
  const int l = (tid - 8) / 16, w = (tid - 8) % 16;
  if (l >= D.L || w > 11 || (w > 8 && !D.qkv_bias)) return false;
  LayerW& L = c->layers[l];
  switch (w) {
    case 0: t->base = (char*)L.g_attn; t->rows = 1; t->cols = D.d; t->gain = true; return true;
    case 1: t->base = (char*)L.qkv; t->rows = D.nq; t->cols = D.d; return true;
    case 2: t->base = (char*)L.qkv; t->rows = D.nkv; t->cols = D.d; t->grp_off = D.nq; return true;
    case 3: t->base = (char*)L.qkv; t->rows = D.nkv; t->cols = D.d; t->grp_off = D.nq + D.nkv; return true;
    case 4: t->base = (char*)L.o; t->rows = D.d; t->cols = D.nq; return true;
    case 5: t->base = (char*)L.g_mlp; t->rows = 1; t->cols = D.d; t->gain = true; return true;
    case 6: t->base = (char*)L.gu; t->rows = D.F; t->cols = D.d; t->grp = 1; t->grp_stride = 2; return true;
    case 7: t->base = (char*)L.gu; t->rows = D.F; t->cols = D.d; t->grp = 1; t->grp_stride = 2; t->grp_off = 1; return true;
    case 8: t->base = (char*)L.dn; t->rows = D.d; t->cols = D.F; return true;
    case 9: t->base = (char*)L.b_qkv; t->rows = 1; t->cols = D.nq; return true;
    case 10: t->base = (char*)L.b_qkv + (size_t)D.nq * D.es; t->rows = 1; t->cols = D.nkv; return true;
    case 11: t->base = (char*)L.b_qkv + (size_t)(D.nq + D.nkv) * D.es; t->rows = 1; t->cols = D.nkv; return true;
  }
  return false;
}

std::vector<int> all_tids(const Dims& D) {
  std::vector<int> v = {0};
  if (!D.tie) v.push_back(1);
  v.push_back(2);
  for (int l = 0; l < D.L; ++l)
    for (int w = 0; w < (D.qkv_bias ? 12 : 9); ++w) v.push_back(8 + 16 * l + w);
  return v;
}

long long dev_row(const TensorLoc& t, long long r) { return (r / t.grp) * t.grp_stride + (r % t.grp) + t.grp_off; }

// Whole tensor between its device rows and a dense host buffer [rows][cols], ordered on stream st
// (the caller synchronises it before using or releasing the host buffer): one strided 2-D copy of
// the full groups of t.grp rows, one more for a partial last group.
cudaError_t copy_tensor(const TensorLoc& t, int es, void* host, cudaMemcpyKind kind, cudaStream_t st) {
  const size_t rb = (size_t)t.cols * es;
  const bool to_dev = kind == cudaMemcpyHostToDevice;
  if (t.grp >= t.rows) {
    char* dev = t.base + (size_t)t.grp_off * rb;
    return to_dev ? cudaMemcpyAsync(dev, host, (size_t)t.rows * rb, kind, st)
                  : cudaMemcpyAsync(host, dev, (size_t)t.rows * rb, kind, st);
  }
  const long long full = t.rows / t.grp, tail = t.rows % t.grp;
  const size_t gw = (size_t)t.grp * rb, dp = (size_t)t.grp_stride * rb;
  char* h = reinterpret_cast<char*>(host);
  char* dev = t.base + (size_t)t.grp_off * rb;
  cudaError_t e = to_dev ? cudaMemcpy2DAsync(dev, dp, h, gw, gw, (size_t)full, kind, st)
                         : cudaMemcpy2DAsync(h, gw, dev, dp, gw, (size_t)full, kind, st);
  if (e != cudaSuccess || tail == 0) return e;
  char* dt = t.base + (size_t)dev_row(t, full * t.grp) * rb;
  char* ht = h + (size_t)full * gw;
  return to_dev ? cudaMemcpyAsync(dt, ht, (size_t)tail * rb, kind, st) : cudaMemcpyAsync(ht, dt, (size_t)tail * rb, kind, st);
}

// Version 1: the header below without the last two fields (a model with neither QKV biases nor
// tied embeddings). Version 2 adds them.
struct FileHeader {
  char magic[4];
  int32_t version, dtype, n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ff, vocab;
  double rms_eps, rope_theta;
  int32_t qkv_bias, tie_embeddings;
};
constexpr size_t kHeaderV1Bytes = offsetof(FileHeader, qkv_bias);

}  // namespace

extern "C" {

jf_status jf_init_random_weights(jf_ctx* c, uint64_t seed, double stdv) {
  if (!c) return JF_EINVAL;
  if (!(stdv >= 0)) return fail(c, JF_EINVAL, "std must be >= 0");
  const Dims& D = c->D;
  for (int tid : all_tids(D)) {
    TensorLoc t;
    tensor_loc(c, tid, &t);
    if (t.gain) {
      CK(launch_fill_f32(reinterpret_cast<float*>(t.base), t.cols, 1.0f, c->st));
      continue;
    }
    const long long grp = t.grp > t.rows ? t.rows : t.grp;
    const long long stride = t.grp > t.rows ? 0 : t.grp_stride;
    CK(launch_init_weights(t.base, D.bf16, t.rows, t.cols, seed, (uint64_t)tid, stdv, grp, stride, t.grp_off, c->st));
  }
  CK(cudaStreamSynchronize(c->st));
  c->weights_ready = true;
  return JF_OK;
}

jf_status jf_get_weights(jf_ctx* c, int tensor_id, long long start, long long count, float* out) {
  if (!c || !out || count < 0 || start < 0) return fail(c, JF_EINVAL, "bad arguments");
  TensorLoc t;
  if (!tensor_loc(c, tensor_id, &t)) return fail(c, JF_EINVAL, "unknown tensor id");
  if (start + count > t.rows * t.cols) return fail(c, JF_EINVAL, "range beyond tensor");
  const int es = t.gain ? 4 : c->D.es;
  std::vector<uint8_t> buf;
  long long done = 0;
  CK(cudaStreamSynchronize(c->st));
  while (done < count) {
    const long long e = start + done;
    const long long r = e / t.cols, col = e % t.cols;
    const long long n = std::min(count - done, t.cols - col);
    buf.resize((size_t)n * es);
    const char* src = t.base + ((size_t)dev_row(t, r) * t.cols + col) * es;
    CK(cudaMemcpy(buf.data(), src, (size_t)n * es, cudaMemcpyDeviceToHost));
    for (long long i = 0; i < n; ++i) {
      if (es == 4) {
        std::memcpy(&out[done + i], &buf[i * 4], 4);
      } else {
        uint16_t b;
        std::memcpy(&b, &buf[i * 2], 2);
        uint32_t u = (uint32_t)b << 16;
        std::memcpy(&out[done + i], &u, 4);
      }
    }
    done += n;
  }
  return JF_OK;
}

jf_status jf_save_weights(jf_ctx* c, const char* path) {
  if (!c || !path) return JF_EINVAL;
  if (!c->weights_ready) return fail(c, JF_ESTATE, "weights not initialised");
  FILE* f = std::fopen(path, "wb");
  if (!f) return fail(c, JF_EIO, "cannot open weight file for writing");
  FileHeader h = {{'J', 'F', 'W', '1'}, 2, c->mc.dtype, c->mc.n_layers, c->mc.d_model, c->mc.n_heads,
                  c->mc.n_kv_heads, c->mc.head_dim, c->mc.d_ff, c->mc.vocab, c->mc.rms_eps, c->mc.rope_theta,
                  c->mc.qkv_bias, c->mc.tie_embeddings};
  bool ok = std::fwrite(&h, sizeof(h), 1, f) == 1;
  CK(cudaStreamSynchronize(c->st));
  std::vector<uint8_t> buf;
  for (int tid : all_tids(c->D)) {
    TensorLoc t;
    tensor_loc(c, tid, &t);
    const int es = t.gain ? 4 : c->D.es;
    buf.resize((size_t)t.rows * t.cols * es);
    if (copy_tensor(t, es, buf.data(), cudaMemcpyDeviceToHost, c->st) != cudaSuccess ||
        cudaStreamSynchronize(c->st) != cudaSuccess) {
      std::fclose(f);
      return fail(c, JF_ECUDA, "copy of weights failed");
    }
    ok = ok && std::fwrite(buf.data(), 1, buf.size(), f) == buf.size();
  }
  ok = (std::fclose(f) == 0) && ok;
  return ok ? JF_OK : fail(c, JF_EIO, "short write of weight file");
}

jf_status jf_load_weights(jf_ctx* c, const char* path) {
  if (!c || !path) return JF_EINVAL;
  FILE* f = std::fopen(path, "rb");
  if (!f) return fail(c, JF_EIO, "cannot open weight file");
  FileHeader h = {};
  bool hdr = std::fread(&h, kHeaderV1Bytes, 1, f) == 1 && std::memcmp(h.magic, "JFW1", 4) == 0 &&
             (h.version == 1 || h.version == 2);
  if (hdr && h.version == 2)
    hdr = std::fread(reinterpret_cast<char*>(&h) + kHeaderV1Bytes, sizeof(h) - kHeaderV1Bytes, 1, f) == 1;
  if (!hdr) {
    std::fclose(f);
    return fail(c, JF_EIO, "not a JFW1 weight file");
  }
  if (h.dtype != c->mc.dtype || h.n_layers != c->mc.n_layers || h.d_model != c->mc.d_model ||
      h.n_heads != c->mc.n_heads || h.n_kv_heads != c->mc.n_kv_heads || h.head_dim != c->mc.head_dim ||
      h.d_ff != c->mc.d_ff || h.vocab != c->mc.vocab || h.qkv_bias != c->mc.qkv_bias ||
      h.tie_embeddings != c->mc.tie_embeddings) {
    std::fclose(f);
    return fail(c, JF_EIO, "weight file has another model shape");
  }
  // read everything first so that a truncated file leaves the context unchanged
  std::vector<std::vector<uint8_t>> data;
  std::vector<TensorLoc> locs;
  for (int tid : all_tids(c->D)) {
    TensorLoc t;
    tensor_loc(c, tid, &t);
    const int es = t.gain ? 4 : c->D.es;
    std::vector<uint8_t> buf((size_t)t.rows * t.cols * es);
    if (std::fread(buf.data(), 1, buf.size(), f) != buf.size()) {
      std::fclose(f);
      return fail(c, JF_EIO, "weight file truncated");
    }
    data.push_back(std::move(buf));
    locs.push_back(t);
  }
  std::fclose(f);
  for (size_t i = 0; i < locs.size(); ++i) {
    const TensorLoc& t = locs[i];
    const int es = t.gain ? 4 : c->D.es;
    CK(copy_tensor(t, es, data[i].data(), cudaMemcpyHostToDevice, c->st));
  }
  CK(cudaStreamSynchronize(c->st));  // the host buffers are released on return
  c->weights_ready = true;
  return JF_OK;
}

// ------------------------------------------------------------------------------------------
// Sequences
// ------------------------------------------------------------------------------------------
jf_status jf_prefill(jf_ctx* c, int seq, const int32_t* prompt, int len, int32_t* next_token) {
  if (!c) return JF_EINVAL;
  if (!c->weights_ready) return fail(c, JF_ESTATE, "weights not initialised");
  if (seq < 0 || seq >= c->D.S || !prompt || len < 1) return fail(c, JF_EINVAL, "bad seq / prompt");
  if (c->h_seq_len[seq] + len > c->D.max_ctx) return fail(c, JF_ECAPACITY, "prompt exceeds max_ctx");
  jf_status s = check_tokens(c, prompt, len);
  if (s != JF_OK) return s;
  return prefill_impl(c, seq, prompt, nullptr, len, next_token);
}

jf_status jf_truncate(jf_ctx* c, int seq, int len) {
  if (!c) return JF_EINVAL;
  if (seq < 0 || seq >= c->D.S || len < 0 || len > c->h_seq_len[seq]) return fail(c, JF_EINVAL, "bad truncate");
  release_pages(c, seq, len);
  return set_seq_len(c, seq, len);
}

jf_status jf_seq_len(jf_ctx* c, int seq, int* out_len) {
  if (!c || !out_len || seq < 0 || seq >= c->D.S) return fail(c, JF_EINVAL, "bad seq");
  *out_len = c->h_seq_len[seq];
  return JF_OK;
}

jf_status jf_jacobi_step(jf_ctx* c, int seq, int n_blocks, const jf_block* blocks, const int32_t* draft,
                         int32_t* accepted_counts, int32_t* committed_tokens, int32_t* n_committed,
                         int32_t* predictions, float* top2) {
  if (!c) return JF_EINVAL;
  const Dims& D = c->D;
  if (!c->weights_ready) return fail(c, JF_ESTATE, "weights not initialised");
  if (seq < 0 || seq >= D.S || n_blocks < 1 || n_blocks > kMaxStepBlocks || !blocks || !draft || !accepted_counts ||
      !committed_tokens || !n_committed)
    return fail(c, JF_EINVAL, "bad arguments");
  const int P = c->h_seq_len[seq];
  if (P < 1) return fail(c, JF_ESTATE, "sequence has no prefix (prefill first)");
  // validate: [RA][PSEUDO...][CAND...], chain positions consecutive from P
  StepBlocks sb = {};
  sb.n_blocks = n_blocks;
  sb.seq = seq;
  sb.P = P;
  int total = 0, chain_end = -1, max_pos = P, max_len = 0;
  bool in_cands = false;
  std::vector<Chain> chains;
  std::vector<int> pos;
  for (int b = 0; b < n_blocks; ++b) {
    const jf_block& bl = blocks[b];
    if (bl.len < 1) return fail(c, JF_EINVAL, "block length must be >= 1");
    if (b == 0) {
      if (bl.kind != JF_BLOCK_RA || bl.start_pos != P || bl.parent != -1)
        return fail(c, JF_EINVAL, "block 0 must be the real-active block at the committed length, parent -1");
      chains.push_back(Chain{seq, 0, bl.len, P});
      chain_end = P + bl.len;
    } else if (bl.kind == JF_BLOCK_PSEUDO) {
      if (in_cands || bl.parent != b - 1 || bl.start_pos != chain_end)
        return fail(c, JF_EINVAL, "a pseudo block must follow the previous main block (parent = previous index)");
      chains[0].nrows += bl.len;
      chain_end += bl.len;
    } else if (bl.kind == JF_BLOCK_CAND) {
      if (bl.parent != -1 || bl.start_pos != P) return fail(c, JF_EINVAL, "a candidate starts at P with parent -1");
      in_cands = true;
      chains.push_back(Chain{seq, total, bl.len, P});
    } else {
      return fail(c, JF_EINVAL, "bad block kind (RA must come first and only once)");
    }
    sb.kind[b] = bl.kind;
    sb.row0[b] = total;
    sb.len[b] = bl.len;
    for (int i = 0; i < bl.len; ++i) pos.push_back(bl.start_pos + i);
    max_pos = std::max(max_pos, bl.start_pos + bl.len);
    if (bl.kind != JF_BLOCK_PSEUDO) max_len = std::max(max_len, bl.len);
    total += bl.len;
    if (total > D.R) return fail(c, JF_ECAPACITY, "more rows than max_rows");
  }
  if ((int)chains.size() > D.max_chains) return fail(c, JF_ECAPACITY, "too many candidates");
  if (max_pos > D.max_ctx) return fail(c, JF_ECAPACITY, "positions beyond max_ctx");
  jf_status s = check_tokens(c, draft, total);
  if (s != JF_OK) return s;
  if ((s = ensure_pages(c, seq, max_pos)) != JF_OK) return s;
  const int nch = (int)chains.size();
  CK(cudaMemcpyAsync(c->tok, draft, (size_t)total * 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->pos, pos.data(), (size_t)total * 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->chains, chains.data(), (size_t)nch * sizeof(Chain), cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->n_chains, &nch, 4, cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->sb_dev, &sb, sizeof(sb), cudaMemcpyHostToDevice, c->st));
  CK(cudaStreamSynchronize(c->st));
  c->chains_bound = nch;
  CK(enqueue_forward(c, total, LM_ARGMAX));
  CK(launch_step_accept(c->sb_dev, c->tok, c->gpred, c->committed_dev, c->commit, c->sres_dev, c->err, c->st));
  CK(launch_commit(c->commit + seq, 1, D.L, c->k_inf, c->v_inf, c->k_pages, c->v_pages,
                   c->page_table + (size_t)seq * D.pps, D.pps, D.n_pages, D.R, D.Hkv, D.hd, D.es, c->seq_len + seq,
                   c->err, c->st));
  StepResult r;
  CK(cudaMemcpyAsync(&r, c->sres_dev, sizeof(r), cudaMemcpyDeviceToHost, c->st));
  if (predictions) CK(cudaMemcpyAsync(predictions, c->gpred, (size_t)total * 4, cudaMemcpyDeviceToHost, c->st));
  if (top2) CK(cudaMemcpyAsync(top2, c->top2, (size_t)total * 8, cudaMemcpyDeviceToHost, c->st));
  CK(cudaStreamSynchronize(c->st));
  if ((s = read_err(c)) != JF_OK) return s;
  if (r.k < 1 || r.k > max_len) return fail(c, JF_EDEVICE, "invalid accepted count");
  CK(cudaMemcpy(committed_tokens, c->committed_dev, (size_t)r.k * 4, cudaMemcpyDeviceToHost));
  for (int b = 0; b < n_blocks; ++b) accepted_counts[b] = r.counts[b];
  *n_committed = r.k;
  c->h_seq_len[seq] = P + r.k;
  return JF_OK;
}

jf_status jf_forward_logits(jf_ctx* c, int seq, int n_rows, const int32_t* tokens, float* logits, float* hidden,
                            int32_t* argmax) {
  if (!c) return JF_EINVAL;
  const Dims& D = c->D;
  if (!c->weights_ready) return fail(c, JF_ESTATE, "weights not initialised");
  if (seq < 0 || seq >= D.S || n_rows < 1 || !tokens) return fail(c, JF_EINVAL, "bad arguments");
  if (logits && n_rows > D.logits_rows) return fail(c, JF_ECAPACITY, "n_rows exceeds logits_rows");
  if (n_rows > D.R) return fail(c, JF_ECAPACITY, "n_rows exceeds max_rows");
  const int P = c->h_seq_len[seq];
  if (P + n_rows > D.max_ctx) return fail(c, JF_ECAPACITY, "positions beyond max_ctx");
  jf_status s = check_tokens(c, tokens, n_rows);
  if (s != JF_OK) return s;
  if ((s = upload_chain(c, seq, P, n_rows, tokens, nullptr)) != JF_OK) return s;
  CK(enqueue_forward(c, n_rows, LM_ARGMAX));
  if (argmax) CK(cudaMemcpyAsync(argmax, c->gpred, (size_t)n_rows * 4, cudaMemcpyDeviceToHost, c->st));
  if (logits) {
    // the LM head again, storing the logits instead of reducing them
    GemmEpi el = {};
    el.kind = EPI_STORE;
    el.y = c->logits;
    el.ldy = D.V;
    CK(gemm(c, c->tm_lm, c->w_lm, c->h, D.V, D.d, n_rows, el, -1));
    CK(cudaMemcpyAsync(logits, c->logits, (size_t)n_rows * D.V * 4, cudaMemcpyDeviceToHost, c->st));
  }
  if (hidden) CK(cudaMemcpyAsync(hidden, c->x, (size_t)n_rows * D.d * 4, cudaMemcpyDeviceToHost, c->st));
  CK(cudaStreamSynchronize(c->st));
  return read_err(c);
}

jf_status jf_generate(jf_ctx* c, int n_seqs, const int32_t* const* prompts, const int32_t* prompt_lens,
                      const jf_gen_params* params, int32_t* out_tokens, jf_gen_stats* stats) {
  if (!c) return JF_EINVAL;
  if (!prompts || !out_tokens) return fail(c, JF_EINVAL, "null prompts / output");
  return generate_impl(c, n_seqs, prompts, nullptr, prompt_lens, params, out_tokens, nullptr, stats, false);
}

jf_status jf_generate_device(jf_ctx* c, int n_seqs, const int32_t* d_prompts, const int32_t* prompt_lens,
                             const jf_gen_params* params, int32_t* d_out_tokens, jf_gen_stats* stats) {
  if (!c) return JF_EINVAL;
  if (!d_prompts || !d_out_tokens) return fail(c, JF_EINVAL, "null prompts / output");
  return generate_impl(c, n_seqs, nullptr, d_prompts, prompt_lens, params, nullptr, d_out_tokens, stats, true);
}

jf_status jf_trajectory_noisy_blocks(const int32_t* traj, int traj_iters, int traj_rows, int seq,
                                     const int32_t* new_tokens, int n_new, int prompt_len, int block_size, int window,
                                     int32_t* noisy_tokens, int32_t* point_index, void* cuda_stream) {
  if (!traj || !new_tokens || !noisy_tokens || !point_index || traj_iters < 0 || traj_rows < 1 || seq < 0 ||
      n_new < 0 || prompt_len < 0 || block_size < 1 || window < 1)
    return JF_EINVAL;
  const int n_blocks = n_new / block_size;
  if (n_blocks == 0) return JF_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(cuda_stream);
  return launch_traj_noisy(traj, traj_iters, traj_rows, seq, new_tokens, prompt_len, block_size, window, n_blocks,
                           noisy_tokens, point_index, st) == cudaSuccess
             ? JF_OK
             : JF_ECUDA;
}

jf_status jf_set_profiling(jf_ctx* c, int enable) {
  if (!c) return JF_EINVAL;
  c->profiling = enable != 0;
  for (int i = 0; i < kProfClasses; ++i) {
    c->prof_ms[i] = 0;
    c->prof_n[i] = 0;
  }
  return JF_OK;
}

jf_status jf_set_wait_limit(jf_ctx* c, uint64_t limit_ns) {
  if (!c) return JF_EINVAL;
  if (limit_ns < kWaitLimitMinNs || limit_ns > kWaitLimitMaxNs)
    return fail(c, JF_EINVAL, "wait limit outside [1 ms, 60 s]");
  if (limit_ns != c->wait_ns) {
    c->wait_ns = limit_ns;
    drop_graphs(c);  // the iteration graphs hold the old limit in their kernel parameters
  }
  return JF_OK;
}

jf_status jf_wait_limit_probe(jf_ctx* c, uint64_t* waited_ns) {
  if (!c) return JF_EINVAL;
  // bytes 8..15 of the error slot receive the time the probe waited
  unsigned long long* waited_dev = reinterpret_cast<unsigned long long*>(c->err + 2);
  CK(launch_wait_probe(c->err, waited_dev, c->wait_ns, c->st));
  c->launches += 1;
  unsigned long long w = 0;
  CK(cudaMemcpyAsync(&w, waited_dev, sizeof(w), cudaMemcpyDeviceToHost, c->st));
  const jf_status s = read_err(c);  // synchronises the stream: the probe has exited
  if (waited_ns) *waited_ns = w;
  return s;
}

jf_status jf_tl_enable(void* records, void* counter) {
#ifdef JF_TIMELINE
  if ((records == nullptr) != (counter == nullptr)) return JF_EINVAL;
  if (jf::tl_set_gemm(records, counter) != cudaSuccess || jf::tl_set_attn(records, counter) != cudaSuccess ||
      jf::tl_set_elem(records, counter) != cudaSuccess || jf::tl_set_decode(records, counter) != cudaSuccess)
    return JF_ECUDA;
  return JF_OK;
#else
  (void)records;
  (void)counter;
  return JF_EUNSUPPORTED;
#endif
}

jf_status jf_kernel_time(jf_ctx* c, int cls, double* total_ms, long long* launches) {
  if (!c || cls < 0 || cls >= kProfClasses || !total_ms || !launches) return fail(c, JF_EINVAL, "bad arguments");
  *total_ms = c->prof_ms[cls];
  *launches = c->prof_n[cls];
  return JF_OK;
}

// ------------------------------------------------------------------------------------------
// Kernel-level entry points (jf_ops.h)
// ------------------------------------------------------------------------------------------
static void op_gemm_shape(int dtype, int N, int K, int M, int k_splits, int* bn, int* nt, int* mt, int* kb, int* sp) {
  *bn = dtype == JF_BF16 ? gemm_bn_for(M) : 32;
  *nt = cdiv(N, kTileN);
  *mt = cdiv(M, *bn);
  *kb = cdiv(K, kTileK);
  if (dtype != JF_BF16) *sp = 1;
  else if (k_splits > 0) *sp = std::min(std::min(k_splits, *kb), 8);
  else *sp = splits_for(*nt, *kb);
}

jf_status jf_op_gemm_workspace_bytes(int N, int K, int M, int k_splits, size_t* out) {
  if (N < 1 || K < 1 || M < 1 || !out) return JF_EINVAL;
  int bn, nt, mt, kb, sp;
  op_gemm_shape(JF_BF16, N, K, M, k_splits, &bn, &nt, &mt, &kb, &sp);
  const size_t partial = sp > 1 ? (size_t)nt * mt * sp * bn * kTileN * 4 : 0;
  *out = rup(partial, 256) + rup((size_t)nt * mt * 4, 256);
  return JF_OK;
}

jf_status jf_op_gemm(int dtype, const void* W, const void* X, float* Y, int N, int K, int M, int k_splits,
                     void* workspace, size_t workspace_bytes, int* err_word, void* cuda_stream) {
  if (dtype != JF_BF16 && dtype != JF_F32) return JF_EINVAL;
  if (!W || !X || !Y || N < 1 || K < 1 || M < 1 || !err_word) return JF_EINVAL;
  if (dtype == JF_BF16) {
    if (K % 8 || ((uintptr_t)W & 15) || ((uintptr_t)X & 15)) return JF_EINVAL;
  }
  int bn, nt, mt, kb, sp;
  op_gemm_shape(dtype, N, K, M, k_splits, &bn, &nt, &mt, &kb, &sp);
  size_t need = 0;
  jf_op_gemm_workspace_bytes(N, K, M, k_splits, &need);
  if (dtype == JF_BF16 && (!workspace || workspace_bytes < need)) return JF_ENOMEM;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(cuda_stream);
  GemmParams p = {};
  p.N = N; p.K = K; p.M = M;
  p.n_tiles = nt; p.m_tiles = mt; p.k_splits = sp; p.kb_total = kb;
  {
    int dev = 0, sms = 152;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    p.grid = sms;
  }
  const size_t partial = sp > 1 ? (size_t)nt * mt * sp * bn * kTileN * 4 : 0;
  p.ws = reinterpret_cast<float*>(workspace);
  p.tile_counter = workspace ? reinterpret_cast<int*>(reinterpret_cast<char*>(workspace) + rup(partial, 256)) : nullptr;
  p.err = err_word;
  p.wait_ns = kWaitLimitDefaultNs;
  p.epi.kind = EPI_STORE;
  p.epi.M = M;
  p.epi.N = N;
  p.epi.y = Y;
  p.epi.ldy = N;
  cudaError_t e;
  if (dtype == JF_BF16) {
    if (gemm_prepare() != cudaSuccess) return JF_ECUDA;  // once per device
    CUtensorMap tA, tB;
    if (!make_tmap(&tA, W, K, N, kTileN) || !make_tmap(&tB, X, K, M, bn)) return JF_ECUDA;
    e = launch_gemm_bf16(tA, tB, p, bn, st);
  } else {
    e = launch_gemm_f32(reinterpret_cast<const float*>(W), reinterpret_cast<const float*>(X), p, st);
  }
  return e == cudaSuccess ? JF_OK : JF_ECUDA;
}

}  // extern "C"
