// Test harness: the decoding state machine of csrc/jf_decode.cu (initial drafts, verification,
// pool, pseudo-accept, tail update, spawn / promote, next rows and chains) compiled for the CPU and
// driven through plain C calls, with the forward pass replaced by predictions the test supplies.
// The kernels' source is included unchanged apart from the edits build.py lists.
#include "jf_decode_host.inc"

#include <map>
#include <utility>
#include <vector>

namespace jf_host {
uint3 thread_idx = {0, 0, 0}, block_idx = {0, 0, 0};
dim3 block_dim(1, 1, 1), grid_dim(1, 1, 1);
static std::vector<int> smem;
int* dyn_smem() { return smem.data(); }

static bool use_script = false;
static std::map<std::pair<int, int>, int> script;

int scripted_inject(const jf::GenCfg& g, int seq, int x, int P0, int it, int* err, inject_fn rule) {
  if (!use_script) return rule(g, seq, x, P0, it, err);
  const int ti = x - P0;
  if (ti < 0 || ti >= g.truth_len) {
    jf_set_error(err, jf::JF_DERR_BOUNDS);
    return 0;
  }
  auto f = script.find({x, it});
  return f != script.end() ? f->second : g.truth[(size_t)seq * g.truth_stride + ti];
}
}  // namespace jf_host

namespace {
std::vector<int> traj_buf;
int traj_counter = 0;
jf::GenCfg G;
std::vector<int> state, tok, pos, out_tokens, iter_log, truth, seqp, late_prompts;
std::vector<jf::Chain> chains;
std::vector<jf::CommitInfo> commit;
jf::IterResult res;
int n_chains_dev = 0, err_word = 0;
}  // namespace

extern "C" {

// seq_n / seq_spawn / join / prompts / prompt_lens: per sequence block size, spawn threshold, join
// iteration (0 = prefilled before the first iteration) and prompt (all prompts concatenated).
int hd_setup(int n, int K, int s_spawn, int pool_size, int Gn, int C, int mode, int init, unsigned long long T,
             unsigned long long seed, int max_new, int eos, int V, int n_seqs, const int* truth_in, int truth_len,
             int max_rows, int max_chains, int max_ctx, const int* seq_n, const int* seq_spawn, const int* join,
             const int* prompts, const int* prompt_lens, int prefill_chunk) {
  if (n_seqs < 1 || n_seqs > jf::kMaxSeqs) return 1;
  const jf::SeqLayout L = jf::seq_layout(n, K, C, Gn, pool_size);
  G = jf::GenCfg{};
  G.n = n; G.K = K; G.s_spawn = s_spawn; G.pool_size = pool_size; G.G = Gn; G.C = C;
  G.mode = mode; G.init = init; G.T = T; G.seed = seed;
  G.max_new = max_new; G.eos = eos; G.V = V; G.n_seqs = n_seqs;
  truth.assign(truth_in, truth_in + (size_t)n_seqs * (truth_len > 0 ? truth_len : 0));
  if (truth.empty()) truth.push_back(0);
  G.truth = truth.data(); G.truth_stride = truth_len; G.truth_len = truth_len;
  G.state_stride = L.total;
  G.max_rows = max_rows; G.max_chains = max_chains; G.max_ctx = max_ctx;
  state.assign((size_t)n_seqs * L.total, 0);
  tok.assign(max_rows, 0);
  pos.assign(max_rows, 0);
  chains.assign(max_chains, jf::Chain{});
  commit.assign(n_seqs, jf::CommitInfo{});
  out_tokens.assign((size_t)n_seqs * max_new, -1);
  iter_log.assign((size_t)max_ctx * n_seqs, -1);
  G.out_tokens = out_tokens.data(); G.iter_log = iter_log.data(); G.max_iters = max_ctx;
  seqp.assign((size_t)n_seqs * jf::kSeqParams, 0);
  late_prompts.clear();
  for (int b = 0; b < n_seqs; ++b) {
    int* sp = &seqp[(size_t)b * jf::kSeqParams];
    sp[jf::SP_N] = seq_n[b];
    sp[jf::SP_SSPAWN] = seq_spawn[b];
    sp[jf::SP_JOIN] = join[b];
    sp[jf::SP_POFF] = (int)late_prompts.size();
    sp[jf::SP_PLEN] = prompt_lens[b];
    long long off = 0;
    for (int c = 0; c < b; ++c) off += prompt_lens[c];
    late_prompts.insert(late_prompts.end(), prompts + off, prompts + off + prompt_lens[b]);
  }
  G.seq_params = seqp.data();
  G.prompts = late_prompts.data();
  G.prefill_chunk = prefill_chunk;
  jf_host::smem.assign((size_t)L.total + max_rows, 0);
  jf_host::use_script = false;
  jf_host::script.clear();
  err_word = 0;
  return 0;
}

// Trajectory record of every iteration (cap iterations of `rows` rows; cap 0 = off); call after hd_setup.
void hd_traj(int cap, int rows) {
  traj_buf.assign((size_t)(cap > 0 ? cap : 1) * (2 + 5 * (size_t)rows), -9);
  traj_counter = 0;
  G.traj = cap > 0 ? traj_buf.data() : nullptr;
  G.traj_cap = cap;
  G.traj_rows = rows;
  G.traj_count = &traj_counter;
}

// Copies the trajectory buffer; returns the number of iterations recorded.
int hd_traj_view(int* out) {
  for (size_t i = 0; i < traj_buf.size(); ++i) out[i] = traj_buf[i];
  return traj_counter;
}

// App. C training points from the trajectory record (k_traj_noisy, one CTA per block run in order as
// one thread): fixed = the sequence's generated tokens.
void hd_traj_noisy(int n_rec, int R, int seq, const int* fixed, int P0, int n, int w, int n_blocks, int* noisy,
                   int* point) {
  std::vector<int> smem_save = jf_host::smem;
  jf_host::smem.assign(64, 0);
  for (int b = 0; b < n_blocks; ++b) {
    jf_host::block_idx.x = b;
    jf::k_traj_noisy(traj_buf.data(), n_rec, R, seq, fixed, P0, n, w, noisy, point);
  }
  jf_host::block_idx.x = 0;
  jf_host::smem = smem_save;
}

// count < 0: the kernels' own injection rule; else (pos[i], it[i]) -> tok[i], truth elsewhere.
void hd_script(int count, const int* p, const int* it, const int* t) {
  jf_host::use_script = count >= 0;
  jf_host::script.clear();
  for (int i = 0; i < count; ++i) jf_host::script[{p[i], it[i]}] = t[i];
}

int hd_init(const int* q0, const int* seq_len, const int* prompt_last) {
  jf::k_gen_init(G, state.data(), q0, seq_len, prompt_last, tok.data(), pos.data(), chains.data(), &n_chains_dev,
                 &res, &err_word);
  return res.next_M;
}

int hd_accept(const int* gpred, int M) {
  jf::k_gen_accept(G, state.data(), gpred, M, tok.data(), pos.data(), chains.data(), &n_chains_dev, commit.data(),
                   &res, &err_word);
  return res.next_M;
}

// rows of the next forward, its chains [n][4] (seq, row0, nrows, pos0), and the iteration's result:
// hdr = (next_M, n_chains, all_done, err); per sequence k, winner, n_out, P; commit [n_seqs][3].
void hd_view(int* tok_out, int* pos_out, int* chains_out, int* hdr, int* k, int* winner, int* n_out, int* P,
             int* commit_out) {
  for (int i = 0; i < res.next_M; ++i) {
    tok_out[i] = tok[i];
    pos_out[i] = pos[i];
  }
  for (int c = 0; c < res.n_chains; ++c) {
    chains_out[4 * c + 0] = chains[c].seq;
    chains_out[4 * c + 1] = chains[c].row0;
    chains_out[4 * c + 2] = chains[c].nrows;
    chains_out[4 * c + 3] = chains[c].pos0;
  }
  hdr[0] = res.next_M;
  hdr[1] = res.n_chains;
  hdr[2] = res.all_done;
  hdr[3] = res.err;
  for (int b = 0; b < G.n_seqs; ++b) {
    k[b] = res.k[b];
    winner[b] = res.winner[b];
    n_out[b] = res.n_out[b];
    P[b] = res.P[b];
    commit_out[3 * b + 0] = commit[b].row0;
    commit_out[3 * b + 1] = commit[b].k;
    commit_out[3 * b + 2] = commit[b].P;
  }
}

void hd_out_tokens(int* out) {
  for (size_t i = 0; i < out_tokens.size(); ++i) out[i] = out_tokens[i];
}

// Step-mode verification (caller-supplied blocks of one sequence): counts[n_blocks], then
// (winner, k, q0_next, err) in out4, the committed tokens in committed[k].
void hd_step(int n_blocks, const int* kind, const int* len, int P, const int* tok_in, const int* gpred, int* counts,
             int* out4, int* committed_out) {
  jf::StepBlocks sb{};
  sb.n_blocks = n_blocks;
  sb.seq = 0;
  sb.P = P;
  int total = 0;
  for (int b = 0; b < n_blocks; ++b) {
    sb.kind[b] = kind[b];
    sb.row0[b] = total;
    sb.len[b] = len[b];
    total += len[b];
  }
  std::vector<jf::CommitInfo> ci(1);
  jf::StepResult r{};
  int e = 0;
  jf::k_step_accept(&sb, tok_in, gpred, committed_out, ci.data(), &r, &e);
  for (int b = 0; b < n_blocks; ++b) counts[b] = r.counts[b];
  out4[0] = r.winner;
  out4[1] = r.k;
  out4[2] = r.q0_next;
  out4[3] = r.err;
}

// The kernels' draft-injection rule for one (seed, threshold, position, iteration, truth token).
int hd_inject_rule(unsigned long long seed, unsigned long long T, int V, int truth_tok, int x, int it) {
  jf::GenCfg g{};
  g.seed = seed; g.T = T; g.V = V;
  g.truth = &truth_tok; g.truth_stride = 1; g.truth_len = 1;
  int e = 0;
  const int r = jf::inject_token_rule(g, 0, x, x, it, &e);
  return e ? -1 : r;
}

}  // extern "C"
