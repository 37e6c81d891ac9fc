/*
 * jf.h -- C ABI of libjf: the Jacobi-decoding hot path of Jacobi Forcing (arXiv 2512.14681)
 * on one NVIDIA GB300 (sm_103a).
 *
 * One Jacobi iteration (Sec. 2.1, Eq. 3; Sec. 3.2 and Algorithm 1 for multi-block decoding and
 * rejection recycling) runs a block of n draft tokens -- or K blocks plus recycled candidates --
 * through ONE forward pass of a causal decoder-only transformer over the exact KV cache of the
 * committed prefix, takes the greedy argmax of every row, accepts the longest fixed-point prefix
 * of the real-active draft (its first token is always correct) and commits that prefix's K/V.
 *
 * Conventions shared by every call:
 *   - Plain pointers and sizes only. "host" pointers are CPU memory, "device" pointers are GPU
 *     memory of the context's device. The caller owns every buffer it passes; the library never
 *     frees caller memory and keeps no pointer to a host buffer after the call returns.
 *   - Device memory: the caller allocates ONE arena of jf_arena_bytes() bytes (e.g. through
 *     PyTorch) and lends it to the context until jf_destroy(). The library allocates no device
 *     memory of its own; it allocates small pinned host buffers for per-iteration results.
 *   - Work is ordered on the caller's CUDA stream (jf_runtime_config.cuda_stream; NULL lets the
 *     library create a non-blocking stream). Calls that return host outputs synchronise it.
 *   - Every call returns a jf_status. Arguments are validated on the host before any launch; a
 *     call that fails validation changes no state. jf_last_error() returns a message for the last
 *     failure. A context is not thread-safe.
 *   - Device-side checks (index bounds, bounded waits of the tensor-core pipeline) report through
 *     an error word read back after each call: JF_EDEVICE / JF_ETIMEOUT. No kernel traps.
 */
#ifndef JF_H
#define JF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  JF_OK = 0,
  JF_EINVAL = 1,        /* invalid argument, shape or call sequence parameter */
  JF_ENOMEM = 2,        /* arena too small, or pinned host allocation failed */
  JF_ECAPACITY = 3,     /* KV pages, rows, sequences or context length exhausted */
  JF_ESTATE = 4,        /* call out of order (e.g. step before prefill, no weights) */
  JF_EIO = 5,           /* weight file missing, truncated or of another shape */
  JF_ECUDA = 6,         /* a CUDA runtime call failed */
  JF_EDEVICE = 7,       /* a kernel found an out-of-range index (bounds check) */
  JF_ETIMEOUT = 8,      /* a bounded device wait gave up */
  JF_EUNSUPPORTED = 9   /* shape not supported by the kernels (see jf_create) */
} jf_status;

typedef enum { JF_F32 = 0, JF_BF16 = 1 } jf_dtype;

/* Decoder shape (Sec. 4.1: the Qwen2.5 family). RMSNorm -> fused QKV (+ per-feature biases when
 * qkv_bias = 1, as in Qwen2.5; added to the projection outputs before the rotary embedding, held in
 * the model dtype) -> rotary embedding
 * (rotate-half pairing, frequency rope_theta^(-2i/head_dim)) -> grouped-query attention ->
 * O projection + residual -> RMSNorm -> SwiGLU MLP + residual; final RMSNorm -> LM head.
 * dtype JF_BF16: weights, KV cache and matrix-product inputs are bf16; accumulation, residual
 * stream, softmax and logits are fp32. JF_F32: everything fp32 (CUDA-core kernels).
 * Supported: head_dim 128 (bf16) or 64/128 (fp32); n_heads*head_dim and n_kv_heads*head_dim
 * multiples of 128; d_model and d_ff multiples of 64; n_heads a multiple of n_kv_heads. */
typedef struct {
  int n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ff, vocab;
  double rms_eps, rope_theta;
  int dtype;
  int qkv_bias;        /* 0 / 1: Q, K and V projections carry per-feature biases */
  int tie_embeddings;  /* 0 / 1: the LM head is the embedding matrix (tensor 1 does not exist) */
} jf_model_config;

/* Capacity. max_rows: in-flight rows per forward (K*n + candidates, or a prefill chunk);
 * max_ctx: positions per sequence (KV pages of 16 tokens are reserved for it; at most 130944
 *   for JF_BF16 models, whose attention stages a sequence's page ids in shared memory);
 * logits_rows: rows jf_forward_logits() may return (0 = that call is unavailable);
 * page_size: tokens per KV page, 0 or 16 (the only size the kernels support; others are
 *   JF_EUNSUPPORTED);
 * max_segments: attention chains one forward may hold, i.e. over all sequences the real-active
 *   draft with its pseudo-active blocks (one chain) plus every verified candidate (one chain each);
 *   0 = min(256, 5 * max_seqs + 1), at most 256. It sizes the attention's lane-state scratch;
 *   calls that would need more return JF_ECAPACITY. */
typedef struct {
  int max_seqs, max_ctx, max_rows, logits_rows;
  void* device_arena;
  size_t arena_bytes;
  void* cuda_stream;
  int page_size;
  int max_segments;
} jf_runtime_config;

typedef struct jf_ctx jf_ctx;

/* Bytes of device arena a context of this shape needs (host-only, no GPU work). */
jf_status jf_arena_bytes(const jf_model_config* model, const jf_runtime_config* rt, size_t* out_bytes);

/* Create a context on the current CUDA device; carves the arena, builds the rotary table. */
jf_status jf_create(const jf_model_config* model, const jf_runtime_config* rt, jf_ctx** out);
void jf_destroy(jf_ctx* ctx);
const char* jf_last_error(const jf_ctx* ctx);

/* Weights. Logical tensors, row-major [out, in]: id 0 embedding [V,d], 1 LM head [V,d] (absent
 * with tie_embeddings), 2 final-norm gain [d]; layer l at 8+16l: +0 attention-norm gain [d],
 * +1 Wq [Hq*hd,d], +2 Wk [Hkv*hd,d], +3 Wv [Hkv*hd,d], +4 Wo [d,Hq*hd], +5 MLP-norm gain [d],
 * +6 W_gate [F,d], +7 W_up [F,d], +8 W_down [d,F], and with qkv_bias +9 b_q [Hq*hd],
 * +10 b_k [Hkv*hd], +11 b_v [Hkv*hd].
 * jf_init_random_weights: every matrix and bias entry = std * N(0,1) from SplitMix64 +
 * Box-Muller keyed by (seed, tensor id, element index), rounded to the model dtype; gains = 1.
 * jf_load_weights / jf_save_weights: raw file "JFW1" (header with the shape, version 2 also with
 * qkv_bias and tie_embeddings; version-1 files load into models with neither), then the existing
 * tensors in id order, matrices and biases in the model dtype, gains fp32).
 * jf_get_weights: copies `count` logical elements of tensor `tensor_id` from `start` into a host
 * fp32 buffer. */
jf_status jf_init_random_weights(jf_ctx* ctx, uint64_t seed, double std);
jf_status jf_load_weights(jf_ctx* ctx, const char* path);
jf_status jf_save_weights(jf_ctx* ctx, const char* path);
jf_status jf_get_weights(jf_ctx* ctx, int tensor_id, long long start, long long count, float* out_host);

/* Prefill (Eq. 1 context x): commit the K/V of `len` prompt tokens (host array) after the
 * sequence's current length, in chunks of max_rows; *next_token (host) = greedy argmax after the
 * last prompt token, i.e. the known-correct first token q0 of the first Jacobi block. */
jf_status jf_prefill(jf_ctx* ctx, int seq, const int32_t* prompt, int len, int32_t* next_token);
jf_status jf_truncate(jf_ctx* ctx, int seq, int len);
jf_status jf_seq_len(jf_ctx* ctx, int seq, int* out_len);

/* One block of a Jacobi step. kind: JF_BLOCK_RA (the real-active draft; exactly one, starting
 * at the committed length P, first token = the known-correct q0), JF_BLOCK_PSEUDO (a
 * pseudo-active block that continues the previous RA/pseudo block: start_pos = its end,
 * parent = its index), JF_BLOCK_CAND (a recycled candidate: start_pos = P, parent = -1). */
typedef enum { JF_BLOCK_RA = 0, JF_BLOCK_PSEUDO = 1, JF_BLOCK_CAND = 2 } jf_block_kind;
typedef struct {
  int kind, start_pos, len, parent;
} jf_block;

/* One Jacobi iteration of sequence `seq` with caller-supplied blocks (Eq. 3; Algorithm 1
 * assemble / forward / verify / cache trim). draft_tokens: host, sum(len) tokens, blocks in
 * order. Outputs (host): accepted_counts[n_blocks] (RA/candidate: 1 + longest run of draft
 * tokens equal to the prediction of the row before them; pseudo: the same run with no free
 * first token); committed_tokens[<= max len] and *n_committed: the winning draft's accepted
 * prefix (largest count, ties to the RA block), whose K/V is committed; predictions[sum(len)]
 * (optional): greedy argmax of every row; top2[sum(len)][2] (optional): fp32 largest and
 * second-largest logit of every row. */
jf_status jf_jacobi_step(jf_ctx* ctx, int seq, int n_blocks, const jf_block* blocks, const int32_t* draft_tokens,
                         int32_t* accepted_counts, int32_t* committed_tokens, int32_t* n_committed,
                         int32_t* predictions, float* top2);

/* Forward of `n_rows` tokens (host) of sequence `seq` at positions P .. P+n_rows-1 with a causal
 * mask, WITHOUT committing: fp32 logits [n_rows][V], final residual stream [n_rows][d] (before
 * the final norm) and argmax [n_rows], each optional (host). n_rows <= logits_rows. */
jf_status jf_forward_logits(jf_ctx* ctx, int seq, int n_rows, const int32_t* tokens, float* logits, float* hidden,
                            int32_t* argmax);

typedef enum { JF_MODE_BLOCK = 0, JF_MODE_WINDOW = 1, JF_MODE_AR = 2 } jf_gen_mode;
typedef enum { JF_INIT_REPEAT = 0, JF_INIT_INJECT = 1 } jf_gen_init;

/* Generation parameters (Eq. 4 block-sequential decoding; running window, Sec. 4.2; Algorithm 1).
 * block_size n; n_blocks K (1 = single block; K > 1 needs JF_MODE_BLOCK); spawn_ratio r (a
 * pseudo block is spawned while fewer than K are active and the newest block has >= ceil(r n)
 * accepted tokens); pool_size / ngram_len G (0 = n) / cand_per_iter: rejection-recycling pool
 * of rejected real-active tails and candidates verified per iteration (pool_size 0 = off);
 * init JF_INIT_REPEAT (free draft positions = the last committed token; Jacobi update
 * thereafter) or JF_INIT_INJECT (free draft positions = truth token, replaced with probability
 * inject_p by another uniform token, keyed by (seed, position, iteration)); truth: greedy
 * continuation of each prompt, [n_seqs][truth_len], required for INJECT with
 * truth_len >= max_new + n_blocks*block_size + G + 1; eos_id -1 = none. */
typedef struct {
  int block_size, n_blocks;
  double spawn_ratio;
  int pool_size, ngram_len, cand_per_iter;
  int mode, init;
  float inject_p;
  uint64_t seed;
  int max_new, eos_id;
  const int32_t* truth;
  int truth_len;
  /* Serving several sequences at once (all optional; NULL / 0 = off). block_sizes (HOST [n_seqs]):
   * block size n_b of sequence b (1 .. block_size, which is then the largest); its spawn threshold
   * is ceil(spawn_ratio * n_b); ignored in JF_MODE_AR. join_iters (HOST [n_seqs]): 0 = the sequence
   * is prefilled before the first iteration; j > 0 = it joins at forward j: its prompt is prefilled
   * inside the decode iterations, prefill_chunk rows (default 64) per forward beside the running
   * sequences' Jacobi rows, and its decoding starts after its last chunk (at once if no other
   * sequence has rows left). max_rows must hold every sequence's rows at once (a joining sequence
   * counts max(its decode rows, prefill_chunk)). */
  const int32_t* block_sizes;
  const int32_t* join_iters;
  int prefill_chunk;
} jf_gen_params;

/* Statistics of one generation. accepted (optional caller buffer [accepted_cap][n_seqs]):
 * tokens committed per iteration (-1 once a sequence is done); rows (optional [accepted_cap]):
 * in-flight rows of each iteration; iter_ms (optional [accepted_cap]): device time of each
 * iteration's graph replay, from CUDA events recorded around it. Times from CUDA events on the
 * context's stream. kernel_launches: libjf kernels launched by the call (prefill, setup and every
 * node of every replayed decode-iteration graph).
 *
 * Jacobi trajectories (Sec. 2.1: the points y^(0), y^(1), ... each block passes through until its
 * fixed point; Sec. 3.1 trains on them). traj (optional, DEVICE int32 buffer lent for the call,
 * traj_cap * (2 + 5 * traj_rows) elements): the device records iteration i < traj_cap at
 * traj + i * (2 + 5 * traj_rows) as [M, i, seq[traj_rows], kind[traj_rows], pos[traj_rows],
 * token[traj_rows], prediction[traj_rows]]: the M rows of that iteration's forward (M <= traj_rows;
 * entries past M are left as they were) with the sequence slot, the kind (0 real-active draft,
 * 1 pseudo-active block, 2 recycled candidate), absolute position, draft token and greedy
 * prediction of each row. traj_rows must be >= n_seqs * (n_blocks * block_size +
 * cand_per_iter * ngram_len) (JF_EINVAL otherwise). traj_iters (out): iterations recorded. Records
 * are written by the acceptance kernel inside the iteration graph; no host copy is made. */
typedef struct {
  int iterations;
  int32_t* accepted;
  int32_t* rows;
  int accepted_cap;
  double prefill_ms, decode_ms;
  long long kernel_launches;
  float* iter_ms;
  int32_t* traj;
  int traj_cap, traj_rows;
  int traj_iters;
} jf_gen_stats;

/* Prefill then Jacobi-decode n_seqs independent sequences (slots 0 .. n_seqs-1, which are reset)
 * until max_new tokens each (or EOS). Host buffers: prompts[i] (prompt_lens[i] tokens),
 * params->truth, out_tokens [n_seqs][max_new] (tokens after an EOS are left as -1). */
jf_status jf_generate(jf_ctx* ctx, int n_seqs, const int32_t* const* prompts, const int32_t* prompt_lens,
                      const jf_gen_params* params, int32_t* out_tokens, jf_gen_stats* stats);

/* Same with device buffers: d_prompts = the prompts concatenated, prompt_lens (HOST array),
 * params->truth a DEVICE pointer [n_seqs][truth_len], d_out_tokens DEVICE [n_seqs][max_new]. */
jf_status jf_generate_device(jf_ctx* ctx, int n_seqs, const int32_t* d_prompts, const int32_t* prompt_lens,
                             const jf_gen_params* params, int32_t* d_out_tokens, jf_gen_stats* stats);

/* Training points from recorded Jacobi trajectories (App. C: for every block, the point of its
 * trajectory whose fraction of unconverged tokens is closest to the block's noise ratio; Eq. 2: the
 * linear progressive schedule t_i = (i mod window) / window over blocks i = 0, 1, ... of the
 * generation). For a generation decoded in JF_MODE_BLOCK with one block of block_size (the setting
 * in which the paper collects trajectories) and recorded into `traj` (jf_gen_stats.traj, traj_iters
 * records of traj_rows rows): block i covers positions prompt_len + i * block_size ...; its points
 * are the records whose first real-active row of sequence `seq` lies in the block (the block's tokens
 * at that iteration: the fixed point before the draft, the draft tokens from there on), then the
 * fixed point itself (index traj_iters). Unconverged = differing from the fixed point, i.e. from
 * new_tokens (the sequence's generated tokens, n_new of them). Ties go to the earlier point. Output
 * for each of the n_new / block_size full blocks: noisy_tokens [blocks][block_size] (the picked
 * point's tokens) and point_index [blocks]. All pointers DEVICE; work is ordered on cuda_stream
 * (no synchronisation). */
jf_status jf_trajectory_noisy_blocks(const int32_t* traj, int traj_iters, int traj_rows, int seq,
                                     const int32_t* new_tokens, int n_new, int prompt_len, int block_size, int window,
                                     int32_t* noisy_tokens, int32_t* point_index, void* cuda_stream);

/* Cumulative device time (ms, CUDA events) and launch count of one kernel class inside
 * jf_generate* decode iterations, when profiling is enabled with jf_set_profiling(ctx, 1) (event
 * records are then placed around every kernel of the iteration graph, which serialises them).
 * kernel_class: 0 = gate/up projection (the largest weight stream), 1 = split-KV attention
 * (partials merged inside the kernel), 2 = all projection GEMMs, 3 = QKV projection,
 * 4 = O projection, 5 = down projection, 6 = LM head + argmax, 7 = reserved (always 0),
 * 8 = RMSNorm, 9 = other (embedding, acceptance, KV commit). jf_set_profiling resets the
 * counters. */
jf_status jf_set_profiling(jf_ctx* ctx, int enable);
jf_status jf_kernel_time(jf_ctx* ctx, int kernel_class, double* total_ms, long long* launches);

/* Bounded device waits. Every wait of a kernel on an asynchronous operation (a TMA copy, a
 * tensor-core MMA, the accumulator hand-over between warps) gives up after the context's wait
 * limit, records the timeout in the context's error word and lets its CTA finish; the call then
 * returns JF_ETIMEOUT and jf_last_error() names the wait. The error word is cleared when it is
 * read, so the context stays usable; the sequences touched by a call that timed out are left as
 * the partial call wrote them (truncate or re-prefill them).
 *
 * jf_set_wait_limit: limit_ns in [1e6, 6e10] (1 ms .. 60 s; default 2 s), for waits launched after
 * the call (the cached decode-iteration graphs are dropped and re-captured). JF_EINVAL outside
 * that range, or for a NULL context.
 *
 * jf_wait_limit_probe: a diagnostic of that error path. Launches one thread on the context's
 * stream that waits, under the context's limit, on a shared-memory mbarrier that nothing arrives
 * at (no copy or MMA is in flight), records the timeout and exits. Synchronises the stream.
 * Returns JF_ETIMEOUT (its expected outcome) and stores the time the wait lasted, in ns, in
 * *waited_ns (NULL: not stored); any other status is a fault of the error path. */
jf_status jf_set_wait_limit(jf_ctx* ctx, uint64_t limit_ns);
jf_status jf_wait_limit_probe(jf_ctx* ctx, uint64_t* waited_ns);

/* Timeline of the forward's kernels, for libraries built with JF_TIMELINE defined (the default
 * build returns JF_EUNSUPPORTED and records nothing). records: device memory for
 * JF_TL_MAX_RECORDS records of 40 bytes {uint32 kernel id, block, SM, pad; uint64 entry time,
 * time past the dependency wait, exit time (ns, %globaltimer)}, written by thread 0 of every CTA;
 * counter: a device int32 the caller zeroes, incremented once per record (records past the
 * maximum are dropped). Kernel ids: 1 RMSNorm, 2 RMSNorm adding split-K partials, 3 QKV finish,
 * 5 attention, 10 + e projection GEMM with epilogue e (13 SwiGLU, 14 argmax, 15 split-K partials),
 * 20 embedding, 21 acceptance, 22 KV commit. (NULL, NULL) stops recording. Not tied to a context:
 * the setting is process-wide and reaches CUDA graphs captured before it. */
#define JF_TL_MAX_RECORDS 2000000
jf_status jf_tl_enable(void* records, void* counter);

#ifdef __cplusplus
}
#endif
#endif /* JF_H */
