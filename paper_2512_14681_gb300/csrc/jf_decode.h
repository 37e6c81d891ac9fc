// Device-side decoding state of libjf (internal; shared by jf_decode.cu and the host runtime).
#pragma once
#include <stdint.h>

#include "jf_internal.h"

namespace jf {

enum GenMode : int { GM_BLOCK = 0, GM_WINDOW = 1 };
enum GenInit : int { GI_REPEAT = 0, GI_INJECT = 1 };

struct GenCfg {
  int n, K, s_spawn, pool_size, G, C, mode, init;  // n: the largest block size (state slot stride)
  unsigned long long T, seed;
  int max_new, eos, V, n_seqs;
  const int* truth;       // [n_seqs][truth_stride] greedy continuation from the prompt end
  int truth_stride, truth_len;
  int state_stride;       // ints per sequence state
  int max_rows, max_chains, max_ctx;
  int* out_tokens;        // [n_seqs][max_new]
  int* iter_log;          // [max_iters][n_seqs] committed count (-1 = inactive)
  int max_iters;
  // Trajectory record (optional, caller-lent device buffer): per iteration i < traj_cap, at
  // traj + i * (2 + 5 * traj_rows): [M, i, seq[traj_rows], kind[traj_rows], pos[traj_rows],
  // token[traj_rows], prediction[traj_rows]] for the M rows of that iteration's forward.
  int* traj;
  int traj_cap, traj_rows;
  int* traj_count;        // device counter of recorded iterations (zeroed by the host per call)
  // Per sequence [n_seqs][kSeqParams]: block size, spawn threshold ceil(r n), join iteration (0 =
  // prefilled before the first iteration; j > 0 = its prompt is prefilled inside the iterations from
  // forward j on, prefill_chunk rows per forward), prompt offset in `prompts`, prompt length.
  const int* seq_params;
  const int* prompts;     // prompts of the sequences that join later (device)
  int prefill_chunk;
};
constexpr int kSeqParams = 5;
enum SeqParam : int { SP_N = 0, SP_SSPAWN, SP_JOIN, SP_POFF, SP_PLEN };
// Phase of a sequence: Jacobi decoding, waiting to join, or prefilling its prompt in chunks.
enum SeqPhase : int { PH_DECODE = 0, PH_WAIT = 1, PH_PREFILL = 2 };

// Layout of one sequence's state (ints). Header fields first.
enum SeqHdr : int {
  H_P = 0, H_Q0, H_NOUT, H_DONE, H_IT, H_LAST, H_NBLK, H_RA_START, H_RA_LEN, H_NCAND, H_POOL_N, H_POOL_HEAD,
  H_P0, H_MAIN_ROW0, H_MAIN_LEN, H_LAST_K, H_WINNER, H_N, H_SSPAWN, H_PHASE, H_JOIN, H_PF, H_PLEN, H_POFF, H_GIT,
  H_COUNT
};

struct SeqLayout {
  int blk_start, blk_na, blk_tok, cand_row0, cand_len, cand_tok, pool, total;
};

__host__ __device__ inline SeqLayout seq_layout(int n, int K, int C, int G, int pool) {
  SeqLayout L;
  int o = H_COUNT;
  L.blk_start = o; o += K;
  L.blk_na = o; o += K;
  L.blk_tok = o; o += K * n;
  L.cand_row0 = o; o += (C > 0 ? C : 1);
  L.cand_len = o; o += (C > 0 ? C : 1);
  L.cand_tok = o; o += (C > 0 ? C : 1) * G;
  L.pool = o; o += (pool > 0 ? pool : 1) * G;
  L.total = (o + 31) & ~31;
  return L;
}

// Per-sequence commit instruction consumed by the KV-commit kernel.
struct CommitInfo {
  int row0, k, P;
};

// Result copied to pinned host memory after every iteration.
struct IterResult {
  int next_M;
  int n_chains;
  int all_done;
  int err;
  int k[kMaxSeqs];
  int n_out[kMaxSeqs];
  int P[kMaxSeqs];
  int winner[kMaxSeqs];
};

// Step mode (caller-supplied blocks of one sequence).
enum BlockKind : int { BK_RA = 0, BK_PSEUDO = 1, BK_CAND = 2 };
constexpr int kMaxStepBlocks = 32;
struct StepBlocks {
  int n_blocks;
  int seq;
  int P;
  int kind[kMaxStepBlocks];
  int row0[kMaxStepBlocks];
  int len[kMaxStepBlocks];
};
struct StepResult {
  int err;
  int winner;
  int k;
  int q0_next;
  int counts[kMaxStepBlocks];
};

cudaError_t launch_gen_init(const GenCfg& g, int* state, const int* q0, const int* seq_len, const int* prompt_last,
                            int* tok, int* pos, Chain* chains, int* n_chains_dev, IterResult* res, int* err,
                            cudaStream_t st);
cudaError_t launch_gen_accept(const GenCfg& g, int* state, const int* gpred, int M_cur, int* tok, int* pos,
                              Chain* chains, int* n_chains_dev, CommitInfo* commit, IterResult* res, int* err, cudaStream_t st);
cudaError_t launch_traj_noisy(const int* traj, int n_rec, int R, int seq, const int* fixed, int P0, int n, int w,
                              int n_blocks, int* noisy, int* point, cudaStream_t st);
cudaError_t launch_step_accept(const StepBlocks* sb, const int* tok, const int* gpred, int* committed,
                               CommitInfo* commit, StepResult* res, int* err, cudaStream_t st);
cudaError_t launch_commit(const CommitInfo* commit, int n_seqs, int L, const void* k_inf, const void* v_inf,
                          void* k_pages, void* v_pages, const int* page_table, int pages_per_seq, int n_pages,
                          int max_rows, int Hkv, int hd, int elem_bytes, int* seq_len, int* err, cudaStream_t st);

}  // namespace jf
