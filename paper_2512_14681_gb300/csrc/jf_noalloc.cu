// jf_op_gemm_noalloc: the bf16 projection GEMM of jf_op_gemm for callers that cannot allocate
// device memory -- code that runs inside a memory allocator's own callbacks, or a process whose
// device memory was fully reserved by another pool before it started -- so it cannot hand the
// kernel a workspace. The split-K scratch (fp32 partial tiles and tile tickets) lives in one fixed
// device array of JF_OP_GEMM_NOALLOC_SCRATCH_BYTES instead.
#include <mutex>

#include "../../include/jf_ops.h"
#include "jf_internal.h"

namespace jf {
cudaError_t gemm_prepare();
}
using namespace jf;

// The shared scratch: every GPU that loads libjf keeps it for the life of the process. In host code
// this name only stands in for the variable; the device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[JF_OP_GEMM_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

size_t rup256(size_t x) { return (x + 255) / 256 * 256; }

// Set-up, once per device, with that device current: the device address of the scratch array.
jf_status scratch_for_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return JF_ECUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return JF_ECUDA;
    g_scratch_ptr[dev] = p;
  }
  // kernel attributes are per device; gemm_prepare sets them once for each device it meets
  if (gemm_prepare() != cudaSuccess) return JF_ECUDA;
  *out = g_scratch_ptr[dev];
  return JF_OK;
}

}  // namespace

extern "C" jf_status jf_op_gemm_noalloc(const void* W, const void* X, float* Y, int N, int K, int M, int k_splits,
                                        int* err_word, void* cuda_stream) {
  if (!W || !X || !Y || !err_word || N < 1 || K < 1 || M < 1) return JF_EINVAL;
  if (K % 8 || ((uintptr_t)W & 15) || ((uintptr_t)X & 15)) return JF_EINVAL;
  size_t need = 0;
  jf_status s = jf_op_gemm_workspace_bytes(N, K, M, k_splits, &need);
  if (s != JF_OK) return s;
  if (need > (size_t)JF_OP_GEMM_NOALLOC_SCRATCH_BYTES) return JF_ECAPACITY;  // too large for the fixed scratch
  void* scratch = nullptr;
  if ((s = scratch_for_current_device(&scratch)) != JF_OK) return s;
  // tile shape and split exactly as jf_op_gemm chooses them
  const int bn = gemm_bn_for(M);
  const int nt = (N + kTileN - 1) / kTileN, mt = (M + bn - 1) / bn, kb = (K + kTileK - 1) / kTileK;
  int sp = k_splits > 0 ? (k_splits < kb ? k_splits : kb) : gemm_default_splits(nt, kb);
  if (sp > 8) sp = 8;
  const size_t partial_bytes = sp > 1 ? (size_t)nt * mt * sp * bn * kTileN * 4 : 0;
  int* tickets = reinterpret_cast<int*>(reinterpret_cast<char*>(scratch) + rup256(partial_bytes));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(cuda_stream);
  // the array keeps the previous call's contents: the tickets must start at zero
  if (cudaMemsetAsync(tickets, 0, (size_t)nt * mt * 4, st) != cudaSuccess) return JF_ECUDA;
  GemmParams p = {};
  p.N = N;
  p.K = K;
  p.M = M;
  p.n_tiles = nt;
  p.m_tiles = mt;
  p.k_splits = sp;
  p.kb_total = kb;
  {
    int dev = 0, sms = 152;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    p.grid = sms;
  }
  p.ws = reinterpret_cast<float*>(scratch);
  p.tile_counter = tickets;
  p.err = err_word;
  p.wait_ns = kWaitLimitDefaultNs;
  p.epi.kind = EPI_STORE;
  p.epi.M = M;
  p.epi.N = N;
  p.epi.y = Y;
  p.epi.ldy = N;
  CUtensorMap tA, tB;
  if (!encode_tmap_bf16(&tA, W, K, N, kTileN) || !encode_tmap_bf16(&tB, X, K, M, bn)) return JF_ECUDA;
  return launch_gemm_bf16(tA, tB, p, bn, st) == cudaSuccess ? JF_OK : JF_ECUDA;
}
