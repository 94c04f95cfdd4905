// Candidate extraction for callers that cannot allocate device memory.
//
// brisk_topk_candidates needs a workspace from its caller. Some callers have
// no way to provide one: a plug-in that runs inside another runtime's process
// and is handed only its input and output buffers, an engine whose memory
// manager has already reserved all of HBM and forbids ad-hoc cudaMalloc, or
// a host that must not allocate on its decode path at all. For them this
// entry point runs the same sweep kernel with its scratch (per-row arrival
// counters and per-chunk partial results) in a fixed array that lives in the
// library itself, so nothing is allocated at call time.
#include <mutex>

#include "brisk_internal.cuh"

using namespace brisk;

namespace {

// Scratch of the no-allocation entry point: 4 MiB in every GPU that loads the
// library, held until the process exits.
constexpr size_t NOALLOC_SCRATCH_BYTES = size_t(4) << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

std::mutex g_noalloc_mu;
std::vector<std::pair<unsigned long long, void*>> g_noalloc_addr;   // (context id, address)

inline size_t up256(size_t x) { return (x + 255) / 256 * 256; }

// Device address of the scratch array in the current CUDA context. The first call in a
// context looks it up (cudaGetSymbolAddress, which also loads the library's module there) and
// caches it under the context's id; a device reset makes a new context with a new id, in which
// the address is looked up again, so a stale address is never used. Host code must never hand
// the array's own name to a kernel, since on the host it is only a stand-in.
void* noalloc_scratch_address() {
  unsigned long long ctx = 0;
  if (!current_context_id(&ctx)) {
    // no context current yet: the lookup below initialises the device's primary context
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return nullptr;
    if (!current_context_id(&ctx)) return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  for (const auto& e : g_noalloc_addr)
    if (e.first == ctx) return e.second;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return nullptr;
  g_noalloc_addr.emplace_back(ctx, p);
  return p;
}

}  // namespace

extern "C" brisk_status brisk_topk_candidates_noalloc(const brisk_dims* d, const void* logits_q,
                                                      int32_t* cand_ids, float* cand_logprob,
                                                      float* lse_q, void* stream) {
  if (brisk_workspace_bytes(d) == 0) return BRISK_ERR_INVALID_ARG;   // dims out of range
  const size_t es = d->logits_dtype == BRISK_DT_BF16 ? 2 : 4;
  if (!logits_q || !cand_ids || !cand_logprob || !lse_q ||
      reinterpret_cast<uintptr_t>(logits_q) % es != 0)
    return BRISK_ERR_INVALID_ARG;
  // scratch layout: status word, arrival counters, per-chunk partial results
  const int rows = d->B * d->L;
  const int nchunk = sweep_chunks(rows, d->V, d->logits_dtype, SWEEP_ROWS);
  const int KP = kp_for(d->K);
  const size_t np = (size_t)rows * nchunk;
  const size_t o_cnt = 256;
  const size_t o_val = o_cnt + up256(sizeof(int32_t) * rows);
  const size_t o_id = o_val + up256(sizeof(float) * np * KP);
  const size_t o_m = o_id + up256(sizeof(int32_t) * np * KP);
  const size_t o_s = o_m + up256(sizeof(float) * np);
  const size_t need = o_s + up256(sizeof(float) * np);
  if (need > NOALLOC_SCRATCH_BYTES) return BRISK_ERR_UNSUPPORTED;   // problem too large for the array

  char* scratch = static_cast<char*>(noalloc_scratch_address());
  if (!scratch) return BRISK_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the array keeps the previous call's contents: the status word and the counters must start at 0
  if (cudaMemsetAsync(scratch, 0, o_val, st) != cudaSuccess) return BRISK_ERR_CUDA;

  SweepLaunch a{};
  SweepSeg& s = a.seg[0];
  s.logits = logits_q;
  s.rows = rows;
  s.kout = d->K;
  s.out_ids = cand_ids;
  s.out_logprob = cand_logprob;
  s.out_lse = lse_q;
  s.counters = reinterpret_cast<int32_t*>(scratch + o_cnt);
  s.part_val = reinterpret_cast<float*>(scratch + o_val);
  s.part_id = reinterpret_cast<int32_t*>(scratch + o_id);
  s.part_m = reinterpret_cast<float*>(scratch + o_m);
  s.part_s = reinterpret_cast<float*>(scratch + o_s);
  a.nseg = 1;
  a.V = d->V;
  a.mode = SWEEP_ROWS;
  a.nchunk = nchunk;
  a.KP = KP;
  a.dtype = d->logits_dtype;
  a.status = reinterpret_cast<int32_t*>(scratch);
  return launch_sweep(a, st) == cudaSuccess ? BRISK_OK : BRISK_ERR_CUDA;
}
