// Verification, KV commit and draft bookkeeping of Jacobi decoding (Algorithm 1 of Jacobi
// Forcing, arXiv 2512.14681; Eq. 3-4 for the single-block case), on the device.
//
// After each forward pass the acceptance kernel, for every sequence:
//   * verifies the real-active (RA) draft and each recycled candidate: k = 1 + the longest run
//     of draft tokens equal to the greedy prediction of the row before them (the first draft
//     token is the known-correct q0); the largest k wins, ties to the RA draft, then to the
//     lower candidate index ("greedy rejection sampling" in the RA block, Sec. 3.2);
//   * records the winner's first k rows for the KV commit (cache trim of Algorithm 1);
//   * pushes the rejected RA tail into the n-gram pool (rejection recycling);
//   * pseudo-accepts each pseudo-active block against the predictions of its chain;
//   * updates drafts: the Jacobi update (next draft = this iteration's predictions) or the
//     draft-injection rule, completes / promotes / spawns blocks, picks the next candidates;
//   * writes the rows and chains of the next forward.
// The commit kernel then copies the accepted rows' K/V of every layer into the KV pages.
#include "jf_decode.h"
#include "jf_device.cuh"

namespace jf {
namespace {

__device__ __forceinline__ uint64_t sm64(uint64_t s, uint64_t i) {
  uint64_t z = s + (i + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Draft-injection rule: the true continuation token at position x, replaced with probability p
// (threshold T = floor(p * 2^53)) by another uniform token, keyed by (seed, x, iteration).
__device__ int inject_token(const GenCfg& g, int seq, int x, int P0, int it, int* err) {
  const int ti = x - P0;
  if (ti < 0 || ti >= g.truth_len) {
    jf_set_error(err, JF_DERR_BOUNDS);
    return 0;
  }
  const int truth = g.truth[(size_t)seq * g.truth_stride + ti];
  const uint64_t s = sm64(g.seed, (uint64_t)x);
  const uint64_t r1 = sm64(s, 2ull * (uint64_t)it);
  if ((r1 >> 11) >= g.T) return truth;
  const uint64_t r2 = sm64(s, 2ull * (uint64_t)it + 1ull);
  return (int)(((uint64_t)truth + 1ull + r2 % (uint64_t)(g.V - 1)) % (uint64_t)g.V);
}

__device__ __forceinline__ int sentinel(int x) { return -(x + 2); }

// thread 0: append pseudo-active blocks while fewer than K are active and the newest block has at
// least s = ceil(r n) accepted tokens.
// Block b of a sequence keeps its n tokens at S[L.blk_tok + b * g.n ..] (g.n: the largest block size).
__device__ void spawn_blocks(const GenCfg& g, const SeqLayout& L, int* S) {
  if (g.K <= 1) return;
  const int n = S[H_N], nst = g.n;
  while (S[H_NBLK] < g.K) {
    const int last = S[H_NBLK] - 1;
    const int start_last = S[L.blk_start + last];
    const int progress = (last == 0) ? (S[H_P] - start_last) : S[L.blk_na + last];
    if (progress < S[H_SSPAWN]) break;
    const int nb = last + 1;
    const int start = start_last + n;
    const int prev_tok = (last == 0) ? S[L.blk_tok + S[H_RA_LEN] - 1] : S[L.blk_tok + last * nst + n - 1];
    S[L.blk_start + nb] = start;
    S[L.blk_na + nb] = 0;
    for (int j = 0; j < n; ++j) S[L.blk_tok + nb * nst + j] = (g.init == GI_INJECT) ? sentinel(start + j) : prev_tok;
    S[H_NBLK] = nb + 1;
  }
}

// thread 0: first drafts of a sequence whose prompt (P tokens) is committed: the RA block
// [q0, fill ...] of its block size, pseudo blocks spawned, empty pool.
__device__ void init_decode(const GenCfg& g, const SeqLayout& L, int* S, int P, int q0, int prompt_last) {
  const int n = S[H_N];
  S[H_PHASE] = PH_DECODE;
  S[H_P] = P;
  S[H_P0] = P;
  S[H_Q0] = q0;
  S[H_LAST] = prompt_last;
  S[H_NBLK] = 1;
  S[L.blk_start] = P;
  S[H_RA_LEN] = n;
  S[L.blk_tok] = q0;
  for (int j = 1; j < n; ++j) S[L.blk_tok + j] = (g.init == GI_INJECT) ? sentinel(P + j) : prompt_last;
  spawn_blocks(g, L, S);
}

// all threads: the rows of the next prefill chunk of a sequence that joined late -- its next
// prompt tokens at the next positions, one causal chain over the committed prefix.
__device__ void finalize_prefill(const GenCfg& g, int* S, int seq, int row_off, int* tok, int* pos, Chain* chains,
                                 int* s_nch, int* s_rows, int* err) {
  const int P = S[H_P], pf = S[H_PF], plen = S[H_PLEN], poff = S[H_POFF];
  const int c = g.prefill_chunk < plen - pf ? g.prefill_chunk : plen - pf;
  const bool fits = c >= 1 && P == pf && row_off + c <= g.max_rows && *s_nch + 1 <= g.max_chains && P + c <= g.max_ctx;
  if (!fits) {
    if (threadIdx.x == 0) {
      jf_set_error(err, JF_DERR_BOUNDS);
      S[H_DONE] = 1;
      *s_rows = 0;
    }
    __syncthreads();
    return;
  }
  for (int j = threadIdx.x; j < c; j += blockDim.x) {
    tok[row_off + j] = g.prompts[poff + pf + j];
    pos[row_off + j] = P + j;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    S[H_MAIN_ROW0] = row_off;
    S[H_MAIN_LEN] = c;
    S[H_RA_LEN] = c;
    S[H_NCAND] = 0;
    chains[*s_nch] = Chain{seq, row_off, c, P};
    *s_nch += 1;
    *s_rows = c;
  }
  __syncthreads();
}

// all threads: resolve injection sentinels, then write this sequence's rows of the next forward
// starting at row_off (thread 0 returns the row count through *s_rows).
__device__ void finalize_seq(const GenCfg& g, const SeqLayout& L, int* S, int seq, int row_off, int* tok, int* pos,
                             Chain* chains, int* s_nch, int* s_rows, int* err) {
  if (S[H_PHASE] == PH_PREFILL) {
    finalize_prefill(g, S, seq, row_off, tok, pos, chains, s_nch, s_rows, err);
    return;
  }
  const int n = S[H_N], nst = g.n;
  const int nblk = S[H_NBLK], Lra = S[H_RA_LEN];
  const int it = S[H_IT], P0 = S[H_P0];
  // sentinels can only be in the RA draft and the pseudo blocks
  const int nslots = Lra + (nblk - 1) * n;
  for (int i = threadIdx.x; i < nslots; i += blockDim.x) {
    int* slot = (i < Lra) ? &S[L.blk_tok + i] : &S[L.blk_tok + (1 + (i - Lra) / n) * nst + (i - Lra) % n];
    const int v = *slot;
    if (v < 0) *slot = inject_token(g, seq, -v - 2, P0, it, err);
  }
  __syncthreads();
  const int P = S[H_P];
  const int mlen = nslots;
  const int nc = S[H_NCAND];
  int total = mlen;
  for (int c = 0; c < nc; ++c) total += S[L.cand_len + c];
  const bool fits = (row_off + total <= g.max_rows) && (*s_nch + 1 + nc <= g.max_chains) &&
                    (P + (nblk > 1 ? (nblk - 1) * n + Lra : Lra) <= g.max_ctx) && (P + g.G <= g.max_ctx || nc == 0);
  if (!fits) {
    if (threadIdx.x == 0) {
      jf_set_error(err, JF_DERR_BOUNDS);
      S[H_DONE] = 1;
      *s_rows = 0;
    }
    __syncthreads();
    return;
  }
  for (int i = threadIdx.x; i < mlen; i += blockDim.x) {
    if (i < Lra) {
      tok[row_off + i] = S[L.blk_tok + i];
      pos[row_off + i] = P + i;
    } else {
      const int bi = 1 + (i - Lra) / n, j = (i - Lra) % n;
      tok[row_off + i] = S[L.blk_tok + bi * nst + j];
      pos[row_off + i] = S[L.blk_start + bi] + j;
    }
  }
  int off = row_off + mlen;
  for (int c = 0; c < nc; ++c) {
    const int cl = S[L.cand_len + c];
    for (int j = threadIdx.x; j < cl; j += blockDim.x) {
      tok[off + j] = S[L.cand_tok + c * g.G + j];
      pos[off + j] = P + j;
    }
    off += cl;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    S[H_MAIN_ROW0] = row_off;
    S[H_MAIN_LEN] = mlen;
    chains[*s_nch] = Chain{seq, row_off, mlen, P};
    *s_nch += 1;
    int o = row_off + mlen;
    for (int c = 0; c < nc; ++c) {
      S[L.cand_row0 + c] = o;
      chains[*s_nch] = Chain{seq, o, S[L.cand_len + c], P};
      *s_nch += 1;
      o += S[L.cand_len + c];
    }
    *s_rows = total;
  }
  __syncthreads();
}

// thread 0: the first waiting sequence (not done) starts its prefill now; -1 if there is none.
__device__ int first_waiting(const GenCfg& g, const int* state) {
  for (int b = 0; b < g.n_seqs; ++b) {
    const int* S = state + (size_t)b * g.state_stride;
    if (!S[H_DONE] && S[H_PHASE] == PH_WAIT) return b;
  }
  return -1;
}

// all threads: when the next forward would have no rows but a sequence still waits to join, that
// sequence starts its prefill in it (a later join iteration cannot be reached without a forward).
__device__ void join_if_idle(const GenCfg& g, int* state, int* S, int* row_off, int* tok, int* pos, Chain* chains,
                             int* s_nch, int* s_rows, int* err, IterResult* res) {
  __shared__ int s_b;
  if (threadIdx.x == 0) s_b = (*row_off == 0) ? first_waiting(g, state) : -1;
  __syncthreads();
  const int b = s_b;
  if (b < 0) return;
  int* Sg = state + (size_t)b * g.state_stride;
  for (int i = threadIdx.x; i < g.state_stride; i += blockDim.x) S[i] = Sg[i];
  __syncthreads();
  if (threadIdx.x == 0) {
    S[H_PHASE] = PH_PREFILL;
    S[H_PF] = 0;
    S[H_P] = 0;
  }
  __syncthreads();
  const SeqLayout L = seq_layout(g.n, g.K, g.C, g.G, g.pool_size);
  finalize_seq(g, L, S, b, *row_off, tok, pos, chains, s_nch, s_rows, err);
  *row_off += *s_rows;
  for (int i = threadIdx.x; i < g.state_stride; i += blockDim.x) Sg[i] = S[i];
  if (threadIdx.x == 0) res->P[b] = S[H_P];
  __syncthreads();
}

// Initial drafts after prefill: RA block [q0, fill...], pseudo blocks spawned, empty pool. A
// sequence with a join iteration j > 0 waits (no rows) until forward j, where its chunked prefill
// starts.
__global__ void k_gen_init(const GenCfg g, int* state, const int* q0, const int* seq_len, const int* prompt_last,
                           int* tok, int* pos, Chain* chains, int* n_chains_dev, IterResult* res, int* err) {
  extern __shared__ int S[];
  __shared__ int s_nch, s_rows;
  pdl_wait();
  const SeqLayout L = seq_layout(g.n, g.K, g.C, g.G, g.pool_size);
  if (threadIdx.x == 0) s_nch = 0;
  int row_off = 0;
  for (int b = 0; b < g.n_seqs; ++b) {
    for (int i = threadIdx.x; i < g.state_stride; i += blockDim.x) S[i] = 0;
    __syncthreads();
    if (threadIdx.x == 0) {
      const int* sp = g.seq_params + (size_t)b * kSeqParams;
      S[H_N] = sp[SP_N];
      S[H_SSPAWN] = sp[SP_SSPAWN];
      S[H_JOIN] = sp[SP_JOIN];
      S[H_POFF] = sp[SP_POFF];
      S[H_PLEN] = sp[SP_PLEN];
      s_rows = 0;
      if (sp[SP_JOIN] <= 0) {
        S[H_PF] = sp[SP_PLEN];
        init_decode(g, L, S, seq_len[b], q0[b], prompt_last[b]);
      } else {
        S[H_PHASE] = PH_WAIT;
      }
    }
    __syncthreads();
    if (S[H_PHASE] != PH_WAIT) {
      finalize_seq(g, L, S, b, row_off, tok, pos, chains, &s_nch, &s_rows, err);
      row_off += s_rows;
    }
    for (int i = threadIdx.x; i < g.state_stride; i += blockDim.x) state[(size_t)b * g.state_stride + i] = S[i];
    if (threadIdx.x == 0) {
      res->k[b] = 0;
      res->n_out[b] = 0;
      res->P[b] = S[H_P];
      res->winner[b] = 0;
    }
    __syncthreads();
  }
  join_if_idle(g, state, S, &row_off, tok, pos, chains, &s_nch, &s_rows, err, res);
  if (threadIdx.x == 0) {
    *n_chains_dev = s_nch;
    res->next_M = row_off;
    res->n_chains = s_nch;
    res->all_done = (row_off == 0);
    res->err = *err;
  }
}

// Jacobi trajectory record (Sec. 2.1: the points y^(0), y^(1), ... a block passes through, each with
// the greedy predictions that give the next one): every row of the forward that just ran, with its
// sequence, kind (0 real-active draft, 1 pseudo-active block, 2 recycled candidate), position, token
// and prediction. Runs before the acceptance step rewrites the rows for the next forward.
__device__ void record_trajectory(const GenCfg& g, const SeqLayout& L, const int* state, const int* gp, int M,
                                  const int* tok, const int* pos) {
  __shared__ int s_it;
  if (threadIdx.x == 0) s_it = *g.traj_count;
  __syncthreads();
  const int it = s_it;
  if (it < g.traj_cap) {
    const int R = g.traj_rows;
    const int Mr = M < R ? M : R;
    int* rec = g.traj + (size_t)it * (2 + 5 * (size_t)R);
    if (threadIdx.x == 0) {
      rec[0] = M;
      rec[1] = it;
    }
    for (int r = threadIdx.x; r < Mr; r += blockDim.x) {
      rec[2 + r] = -1;
      rec[2 + R + r] = -1;
      rec[2 + 2 * R + r] = pos[r];
      rec[2 + 3 * R + r] = tok[r];
      rec[2 + 4 * R + r] = gp[r];
    }
    __syncthreads();
    for (int b = 0; b < g.n_seqs; ++b) {
      const int* S = state + (size_t)b * g.state_stride;
      if (S[H_DONE]) continue;  // a finished sequence has no rows in this forward
      if (S[H_PHASE] == PH_WAIT) continue;  // nor does one still waiting to join
      const int mr0 = S[H_MAIN_ROW0], mlen = S[H_MAIN_LEN], lra = S[H_RA_LEN];
      const bool prefill = S[H_PHASE] == PH_PREFILL;
      for (int r = threadIdx.x; r < mlen; r += blockDim.x) {
        const int row = mr0 + r;
        if (row >= 0 && row < Mr) {
          rec[2 + row] = b;
          rec[2 + R + row] = prefill ? 3 : (r < lra ? 0 : 1);
        }
      }
      const int nc = S[H_NCAND];
      for (int c = 0; c < nc; ++c) {
        const int cr0 = S[L.cand_row0 + c], cl = S[L.cand_len + c];
        for (int r = threadIdx.x; r < cl; r += blockDim.x) {
          const int row = cr0 + r;
          if (row >= 0 && row < Mr) {
            rec[2 + row] = b;
            rec[2 + R + row] = 2;
          }
        }
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *g.traj_count = it + 1;
}

__global__ void k_gen_accept(const GenCfg g, int* state, const int* gpred, int M_cur, int* tok, int* pos,
                             Chain* chains, int* n_chains_dev, CommitInfo* commit, IterResult* res, int* err) {
  extern __shared__ int sm[];
  int* S = sm;
  int* gp = sm + g.state_stride;  // predictions of the current forward
  __shared__ int s_nch, s_rows;
  JF_TL_ENTRY();
  pdl_wait();
  JF_TL_WAITED();
  const SeqLayout L = seq_layout(g.n, g.K, g.C, g.G, g.pool_size);
  for (int i = threadIdx.x; i < M_cur; i += blockDim.x) gp[i] = gpred[i];
  if (threadIdx.x == 0) s_nch = 0;
  __syncthreads();
  if (g.traj) record_trajectory(g, L, state, gp, M_cur, tok, pos);
  const int nst = g.n, G = g.G;
  int row_off = 0;
  int all_done = 1;
  for (int b = 0; b < g.n_seqs; ++b) {
    int* Sg = state + (size_t)b * g.state_stride;
    for (int i = threadIdx.x; i < g.state_stride; i += blockDim.x) S[i] = Sg[i];
    __syncthreads();
    const bool was_done = S[H_DONE] != 0;
    if (threadIdx.x == 0) {
      commit[b] = CommitInfo{0, 0, S[H_P]};
      const int git = S[H_GIT];
      S[H_GIT] = git + 1;
      if (!was_done && S[H_PHASE] == PH_WAIT) {
        // a late sequence joins: its first prefill chunk rides in the next forward
        if (git + 1 >= S[H_JOIN]) {
          S[H_PHASE] = PH_PREFILL;
          S[H_PF] = 0;
          S[H_P] = 0;
        }
      } else if (!was_done && S[H_PHASE] == PH_PREFILL) {
        // a prefill chunk ran: all its rows are committed; after the last one, decoding starts
        const int mr0 = S[H_MAIN_ROW0], c = S[H_MAIN_LEN], P = S[H_P];
        commit[b] = CommitInfo{mr0, c, P};
        S[H_PF] += c;
        S[H_P] = P + c;
        S[H_LAST_K] = 0;
        S[H_WINNER] = 0;
        if (S[H_PF] >= S[H_PLEN])
          init_decode(g, L, S, P + c, gp[mr0 + c - 1], g.prompts[S[H_POFF] + S[H_PLEN] - 1]);
      } else if (!was_done) {
        const int n = S[H_N];
        const int P = S[H_P], Lra = S[H_RA_LEN], mr0 = S[H_MAIN_ROW0], mlen = S[H_MAIN_LEN];
        const int nblk = S[H_NBLK];
        int* ra = S + L.blk_tok;
        // verification of the RA draft and of each candidate
        int k_ra = 1;
        while (k_ra < Lra && ra[k_ra] == gp[mr0 + k_ra - 1]) ++k_ra;
        int win = 0, k = k_ra, wr0 = mr0, wlen = Lra;
        const int* wt = ra;
        for (int c = 0; c < S[H_NCAND]; ++c) {
          const int* ct = S + L.cand_tok + c * G;
          const int cr0 = S[L.cand_row0 + c], cl = S[L.cand_len + c];
          int kc = 1;
          while (kc < cl && ct[kc] == gp[cr0 + kc - 1]) ++kc;
          if (kc > k) {
            win = c + 1;
            k = kc;
            wr0 = cr0;
            wlen = cl;
            wt = ct;
          }
        }
        commit[b] = CommitInfo{wr0, k, P};
        // committed tokens (stop at max_new or EOS)
        int nout = S[H_NOUT], last = S[H_LAST], done = 0;
        for (int i = 0; i < k && !done; ++i) {
          g.out_tokens[(size_t)b * g.max_new + nout] = wt[i];
          ++nout;
          last = wt[i];
          if (nout >= g.max_new || wt[i] == g.eos) done = 1;
        }
        const int new_q0 = gp[wr0 + k - 1];
        const int Pn = P + k;
        // rejection recycling: the rejected RA tail, padded with the following in-flight tokens
        if (g.pool_size > 0 && k_ra < Lra) {
          int pn = S[H_POOL_N], ph = S[H_POOL_HEAD], slot;
          if (pn < g.pool_size) {
            slot = (ph + pn) % g.pool_size;
            S[H_POOL_N] = pn + 1;
          } else {
            slot = ph;
            S[H_POOL_HEAD] = (ph + 1) % g.pool_size;
          }
          int prev = 0;
          for (int j = 0; j < G; ++j) {
            const int idx = k_ra + j;
            int tv;
            if (idx < mlen) {
              tv = (idx < Lra) ? ra[idx] : S[L.blk_tok + (1 + (idx - Lra) / n) * nst + (idx - Lra) % n];
            } else {
              tv = prev;
            }
            S[L.pool + slot * G + j] = tv;
            prev = tv;
          }
        }
        // pseudo-active blocks: pseudo-accept against the main chain's predictions
        for (int bi = 1; bi < nblk; ++bi) {
          const int start = S[L.blk_start + bi];
          int na = S[L.blk_na + bi];
          int* bt = S + L.blk_tok + bi * nst;
          while (na < n && bt[na] == gp[mr0 + (start + na - 1 - P)]) ++na;
          S[L.blk_na + bi] = na;
          for (int x = start + na; x < start + n; ++x)
            bt[x - start] = (g.init == GI_INJECT) ? sentinel(x) : gp[mr0 + (x - 1 - P)];
        }
        // header
        S[H_Q0] = new_q0;
        S[H_P] = Pn;
        S[H_NOUT] = nout;
        S[H_DONE] = done;
        S[H_LAST] = last;
        S[H_LAST_K] = k;
        S[H_WINNER] = win;
        const int it_old = S[H_IT];
        S[H_IT] = it_old + 1;
        if (g.iter_log && it_old < g.max_iters) g.iter_log[(size_t)it_old * g.n_seqs + b] = k;
        // RA tail update / block completion / promotion
        const int ra_start = S[L.blk_start];
        auto tail_pred = [&](int x, int fallback) -> int {
          const int r = x - 1 - P;
          if (r >= 0 && r < wlen) return gp[wr0 + r];
          if (x - 1 < P + mlen) return gp[mr0 + (x - 1 - P)];
          return fallback;
        };
        int Ln;
        if (g.mode == GM_WINDOW) {
          S[L.blk_start] = Pn;
          Ln = n;
          ra[0] = new_q0;
          for (int x = Pn + 1; x < Pn + n; ++x) ra[x - Pn] = (g.init == GI_INJECT) ? sentinel(x) : tail_pred(x, last);
        } else if (Pn >= ra_start + n) {
          if (nblk > 1) {
            for (int j = 0; j < n; ++j) ra[j] = S[L.blk_tok + nst + j];
            ra[0] = new_q0;
            S[L.blk_start] = S[L.blk_start + 1];
            for (int bi = 1; bi + 1 < nblk; ++bi) {
              S[L.blk_start + bi] = S[L.blk_start + bi + 1];
              S[L.blk_na + bi] = S[L.blk_na + bi + 1];
              for (int j = 0; j < n; ++j) S[L.blk_tok + bi * nst + j] = S[L.blk_tok + (bi + 1) * nst + j];
            }
            S[H_NBLK] = nblk - 1;
          } else {
            S[L.blk_start] = Pn;
            ra[0] = new_q0;
            for (int x = Pn + 1; x < Pn + n; ++x) ra[x - Pn] = (g.init == GI_INJECT) ? sentinel(x) : last;
          }
          Ln = n;
        } else {
          Ln = ra_start + n - Pn;
          ra[0] = new_q0;
          for (int x = Pn + 1; x < ra_start + n; ++x)
            ra[x - Pn] = (g.init == GI_INJECT) ? sentinel(x) : tail_pred(x, last);
        }
        S[H_RA_LEN] = Ln;
        spawn_blocks(g, L, S);
        // recycled candidates for the next iteration: keys equal to q0 first, most recent first
        int cnt = 0;
        if (g.pool_size > 0 && g.C > 0 && Ln >= 2) {
          const int pn = S[H_POOL_N], ph = S[H_POOL_HEAD];
          const int clen = G < Ln ? G : Ln;
          for (int pass = 0; pass < 2 && cnt < g.C; ++pass)
            for (int i = pn - 1; i >= 0 && cnt < g.C; --i) {
              const int slot = (ph + i) % g.pool_size;
              const int* ent = S + L.pool + slot * G;
              if ((ent[0] == new_q0) != (pass == 0)) continue;
              int* ct = S + L.cand_tok + cnt * G;
              ct[0] = new_q0;
              for (int j = 1; j < clen; ++j) ct[j] = ent[j];
              S[L.cand_len + cnt] = clen;
              ++cnt;
            }
        }
        S[H_NCAND] = cnt;
      }
    }
    __syncthreads();
    if (!S[H_DONE] && S[H_PHASE] != PH_WAIT) {
      finalize_seq(g, L, S, b, row_off, tok, pos, chains, &s_nch, &s_rows, err);
      row_off += s_rows;
    }
    for (int i = threadIdx.x; i < g.state_stride; i += blockDim.x) Sg[i] = S[i];
    if (threadIdx.x == 0) {
      if (!S[H_DONE]) all_done = 0;
      res->k[b] = was_done ? 0 : S[H_LAST_K];
      res->n_out[b] = S[H_NOUT];
      res->P[b] = S[H_P];
      res->winner[b] = S[H_WINNER];
    }
    __syncthreads();
  }
  join_if_idle(g, state, S, &row_off, tok, pos, chains, &s_nch, &s_rows, err, res);
  if (threadIdx.x == 0) {
    *n_chains_dev = s_nch;
    res->next_M = row_off;
    res->n_chains = s_nch;
    res->all_done = all_done;
    res->err = *err;
  }
  JF_TL_EXIT(TL_ACCEPT);
  pdl_launch_dependents();
}

// Training points from the recorded trajectories (App. C with the linear progressive schedule of
// Eq. 2). Block i of sequence `seq` covers positions P0 + i n .. + n - 1; its trajectory points are
// the records whose first real-active row of the sequence lies in the block (the block's tokens at
// that iteration: the fixed point before the draft, the draft from there on), then the fixed point
// itself (index n_rec). The pick is the point whose number u of unconverged tokens (positions that
// differ from the fixed point) minimises |u w - (i mod w) n| = n w |u / n - t_i|, the earlier point
// on a tie (blocks counted from 0, so t rises from 0 within each window of w blocks). One CTA per
// block; `fixed` = the sequence's generated tokens.
__global__ void k_traj_noisy(const int* traj, int n_rec, int R, int seq, const int* fixed, int P0, int n, int w,
                             int* noisy, int* point) {
  extern __shared__ int sm[];
  long long* s_key = reinterpret_cast<long long*>(sm);  // [blockDim.x] best (distance, index) per thread
  const int i = blockIdx.x;
  const int b0 = P0 + i * n;
  const long long target = (long long)(i % w) * n;
  const size_t stride = 2 + 5 * (size_t)R;
  long long best = (target << 32) | (long long)n_rec;  // the fixed point: u = 0
  for (int j = threadIdx.x; j < n_rec; j += blockDim.x) {
    const int* rec = traj + (size_t)j * stride;
    const int M = rec[0] < R ? rec[0] : R;
    int p_ra = -1, u = 0;
    for (int r = 0; r < M; ++r) {
      if (rec[2 + r] != seq || rec[2 + R + r] != 0) continue;
      const int x = rec[2 + 2 * R + r];
      if (p_ra < 0) p_ra = x;
      if (x >= b0 && x < b0 + n && rec[2 + 3 * R + r] != fixed[x - P0]) ++u;
    }
    if (p_ra < b0 || p_ra >= b0 + n) continue;
    const long long d = (long long)u * w - target;
    const long long key = ((d < 0 ? -d : d) << 32) | (long long)j;
    if (key < best) best = key;
  }
  s_key[threadIdx.x] = best;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int t = 1; t < (int)blockDim.x; ++t)
      if (s_key[t] < best) best = s_key[t];
    s_key[0] = best;
    point[i] = (int)(best & 0xffffffffLL);
  }
  __syncthreads();
  const int jb = (int)(s_key[0] & 0xffffffffLL);
  for (int x = threadIdx.x; x < n; x += blockDim.x) noisy[(size_t)i * n + x] = fixed[i * n + x];
  __syncthreads();
  if (jb < n_rec) {
    const int* rec = traj + (size_t)jb * stride;
    const int M = rec[0] < R ? rec[0] : R;
    for (int r = threadIdx.x; r < M; r += blockDim.x) {
      if (rec[2 + r] != seq || rec[2 + R + r] != 0) continue;
      const int x = rec[2 + 2 * R + r];
      if (x >= b0 && x < b0 + n) noisy[(size_t)i * n + (x - b0)] = rec[2 + 3 * R + r];
    }
  }
}

// Step mode: blocks supplied by the caller for one sequence.
__global__ void k_step_accept(const StepBlocks* sbp, const int* tok, const int* gpred, int* committed,
                              CommitInfo* commit, StepResult* res, int* err) {
  pdl_wait();
  if (threadIdx.x != 0) return;
  const StepBlocks& sb = *sbp;
  int win = -1, k = 0, wr0 = 0;
  for (int b = 0; b < sb.n_blocks; ++b) {
    const int r0 = sb.row0[b], len = sb.len[b];
    int c;
    if (sb.kind[b] == BK_PSEUDO) {
      c = 0;
      while (c < len && tok[r0 + c] == gpred[r0 + c - 1]) ++c;
    } else {
      c = 1;
      while (c < len && tok[r0 + c] == gpred[r0 + c - 1]) ++c;
      if (c > k) {
        k = c;
        win = b;
        wr0 = r0;
      }
    }
    res->counts[b] = c;
  }
  for (int i = 0; i < k; ++i) committed[i] = tok[wr0 + i];
  commit[sb.seq] = CommitInfo{wr0, k, sb.P};
  res->winner = win;
  res->k = k;
  res->q0_next = k > 0 ? gpred[wr0 + k - 1] : -1;
  res->err = *err;
}

// Copy the accepted rows' K/V of layer blockIdx.x, sequence blockIdx.y into the KV pages.
__global__ void k_commit(const CommitInfo* commit, const uint8_t* k_inf, const uint8_t* v_inf, uint8_t* k_pages,
                         uint8_t* v_pages, const int* page_table, int pages_per_seq, int n_pages, int max_rows, int Hkv,
                         int hd, int es, int* seq_len, int* err) {
  JF_TL_ENTRY();
  pdl_wait();
  JF_TL_WAITED();
  const int l = blockIdx.x, b = blockIdx.y;
  const CommitInfo ci = commit[b];
  const size_t head_bytes = (size_t)hd * es;
  const size_t row_bytes = (size_t)Hkv * head_bytes;
  const int vec_per_row = (int)(row_bytes / 16);
  const int vec_per_head = (int)(head_bytes / 16);
  const uint8_t* ksrc = k_inf + (size_t)l * max_rows * row_bytes;
  const uint8_t* vsrc = v_inf + (size_t)l * max_rows * row_bytes;
  for (int i = threadIdx.x; i < ci.k * vec_per_row; i += blockDim.x) {
    const int j = i / vec_per_row, v = i % vec_per_row;
    const int p = ci.P + j;
    const int page = page_table[(size_t)b * pages_per_seq + (p >> 4)];
    if (page < 0 || page >= n_pages) {
      jf_set_error(err, JF_DERR_BOUNDS);
      continue;
    }
    const int h = v / vec_per_head, w = v % vec_per_head;
    const size_t dst = ((((size_t)l * n_pages + page) * Hkv + h) * kPage + (p & 15)) * head_bytes + (size_t)w * 16;
    const size_t src = (size_t)(ci.row0 + j) * row_bytes + (size_t)v * 16;
    *reinterpret_cast<uint4*>(k_pages + dst) = *reinterpret_cast<const uint4*>(ksrc + src);
    *reinterpret_cast<uint4*>(v_pages + dst) = *reinterpret_cast<const uint4*>(vsrc + src);
  }
  if (l == 0 && threadIdx.x == 0) seq_len[b] = ci.P + ci.k;
  JF_TL_EXIT(TL_COMMIT);
  pdl_launch_dependents();
}

cudaLaunchConfig_t pdl_cfg(dim3 grid, dim3 block, size_t smem, cudaStream_t st, cudaLaunchAttribute* at) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cfg;
}

}  // namespace

#ifdef JF_TIMELINE
JF_TL_SETTER(tl_set_decode)
#endif

cudaError_t launch_gen_init(const GenCfg& g, int* state, const int* q0, const int* seq_len, const int* prompt_last,
                            int* tok, int* pos, Chain* chains, int* n_chains_dev, IterResult* res, int* err,
                            cudaStream_t st) {
  const size_t smem = (size_t)g.state_stride * 4;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_gen_init, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  k_gen_init<<<1, 256, smem, st>>>(g, state, q0, seq_len, prompt_last, tok, pos, chains, n_chains_dev, res, err);
  return cudaGetLastError();
}

cudaError_t launch_gen_accept(const GenCfg& g, int* state, const int* gpred, int M_cur, int* tok, int* pos,
                              Chain* chains, int* n_chains_dev, CommitInfo* commit, IterResult* res, int* err,
                              cudaStream_t st) {
  const size_t smem = ((size_t)g.state_stride + (size_t)g.max_rows) * 4;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_gen_accept, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchAttribute at[1];
  cudaLaunchConfig_t cfg = pdl_cfg(dim3(1), dim3(256), smem, st, at);
  return cudaLaunchKernelEx(&cfg, k_gen_accept, g, state, gpred, M_cur, tok, pos, chains, n_chains_dev, commit, res,
                            err);
}

cudaError_t launch_traj_noisy(const int* traj, int n_rec, int R, int seq, const int* fixed, int P0, int n, int w,
                              int n_blocks, int* noisy, int* point, cudaStream_t st) {
  constexpr int kThreads = 128;
  k_traj_noisy<<<n_blocks, kThreads, kThreads * sizeof(long long), st>>>(traj, n_rec, R, seq, fixed, P0, n, w, noisy,
                                                                         point);
  return cudaGetLastError();
}

cudaError_t launch_step_accept(const StepBlocks* sb, const int* tok, const int* gpred, int* committed,
                               CommitInfo* commit, StepResult* res, int* err, cudaStream_t st) {
  cudaLaunchAttribute at[1];
  cudaLaunchConfig_t cfg = pdl_cfg(dim3(1), dim3(32), 0, st, at);
  return cudaLaunchKernelEx(&cfg, k_step_accept, sb, tok, gpred, committed, commit, res, err);
}

cudaError_t launch_commit(const CommitInfo* commit, int n_seqs, int L, const void* k_inf, const void* v_inf,
                          void* k_pages, void* v_pages, const int* page_table, int pages_per_seq, int n_pages,
                          int max_rows, int Hkv, int hd, int elem_bytes, int* seq_len, int* err, cudaStream_t st) {
  cudaLaunchAttribute at[1];
  cudaLaunchConfig_t cfg = pdl_cfg(dim3(L, n_seqs), dim3(256), 0, st, at);
  return cudaLaunchKernelEx(&cfg, k_commit, commit, reinterpret_cast<const uint8_t*>(k_inf),
                            reinterpret_cast<const uint8_t*>(v_inf), reinterpret_cast<uint8_t*>(k_pages),
                            reinterpret_cast<uint8_t*>(v_pages), page_table, pages_per_seq, n_pages, max_rows, Hkv,
                            hd, elem_bytes, seq_len, err);
}

}  // namespace jf
