// Internal declarations shared by the CUDA translation units of the decode tail.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <math.h>
#include <atomic>
#include <mutex>
#include <utility>
#include <vector>

#include "../../include/brisk.h"

namespace brisk {

constexpr unsigned FULL_MASK = 0xffffffffu;
constexpr float LOG2E = 1.4426950408889634f;   // log2(e): exp(x) = 2^(x log2 e)
constexpr float LN2 = 0.6931471805599453f;
constexpr int INVALID_ID = 0x7fffffff;
constexpr float RESID_Z_FLOOR = 1e-6f;         // residual mass below which the verifier argmax is used

// ---------------------------------------------------------------- element access
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> struct Vec;   // 16-byte vector of T
template <> struct Vec<float> { static constexpr int N = 4; };
template <> struct Vec<__nv_bfloat16> { static constexpr int N = 8; };

// Streaming 16-byte load that skips L1 allocation (each logit is read once).
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
  return r;
}

__device__ __forceinline__ void unpack(const uint4& w, float (&f)[8], __nv_bfloat16) {
  const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    f[2 * j] = __uint_as_float(u[j] << 16);
    f[2 * j + 1] = __uint_as_float(u[j] & 0xffff0000u);
  }
}
__device__ __forceinline__ void unpack(const uint4& w, float (&f)[4], float) {
  f[0] = __uint_as_float(w.x);
  f[1] = __uint_as_float(w.y);
  f[2] = __uint_as_float(w.z);
  f[3] = __uint_as_float(w.w);
}

// Hardware base-2 exponential (MUFU), flushes subnormal results to zero.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---------------------------------------------------------------- ordering
// Candidate order of the method: logit descending, then id ascending.
__device__ __forceinline__ bool better(float v1, int i1, float v2, int i2) {
  return v1 > v2 || (v1 == v2 && i1 < i2);
}

// Insert (v, id) into a list sorted best-first; the worst entry falls off.
template <int KP>
__device__ __forceinline__ void list_insert(float v, int id, float (&vals)[KP], int (&ids)[KP]) {
#pragma unroll
  for (int j = 0; j < KP; ++j) {
    const bool sw = better(v, id, vals[j], ids[j]);
    const float tv = vals[j];
    const int ti = ids[j];
    vals[j] = sw ? v : tv;
    ids[j] = sw ? id : ti;
    v = sw ? tv : v;
    id = sw ? ti : id;
  }
}

template <int KP>
__device__ __forceinline__ void list_clear(float (&vals)[KP], int (&ids)[KP]) {
#pragma unroll
  for (int j = 0; j < KP; ++j) {
    vals[j] = -INFINITY;
    ids[j] = INVALID_ID;
  }
}

// Warp-wide extraction of the best `kout` entries of 32 sorted lists. Lane r < kout ends
// holding the r-th best in (out_v, out_i).
template <int KP>
__device__ __forceinline__ void warp_extract(float (&vals)[KP], int (&ids)[KP], int kout,
                                             float& out_v, int& out_i) {
  const int lane = threadIdx.x & 31;
  out_v = -INFINITY;
  out_i = INVALID_ID;
  for (int r = 0; r < kout; ++r) {
    float bv = vals[0];
    int bi = ids[0];
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      const float ov = __shfl_xor_sync(FULL_MASK, bv, off);
      const int oi = __shfl_xor_sync(FULL_MASK, bi, off);
      if (better(ov, oi, bv, bi)) {
        bv = ov;
        bi = oi;
      }
    }
    const bool win = (ids[0] == bi) && (vals[0] == bv);
#pragma unroll
    for (int j = 0; j < KP - 1; ++j) {
      vals[j] = win ? vals[j + 1] : vals[j];
      ids[j] = win ? ids[j + 1] : ids[j];
    }
    if (win) {
      vals[KP - 1] = -INFINITY;
      ids[KP - 1] = INVALID_ID;
    }
    if (lane == r) {
      out_v = bv;
      out_i = bi;
    }
  }
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int off = 16; off; off >>= 1) x += __shfl_xor_sync(FULL_MASK, x, off);
  return x;
}
__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int off = 16; off; off >>= 1) x = fmaxf(x, __shfl_xor_sync(FULL_MASK, x, off));
  return x;
}

// Combine per-lane (max, sum of exp(x - max)) pairs into the warp's pair.
__device__ __forceinline__ void warp_lse_combine(float& m, float& s) {
  const float M = warp_max(m);
  float t = (m == -INFINITY) ? 0.f : s * ex2((m - M) * LOG2E);
  t = warp_sum(t);
  m = M;
  s = t;
}

// Shared-memory carveouts (KB) the kernels ask for. An SM cannot change its L1/shared split
// while a CTA is resident, and the first kernel to land on an idle SM sets it, so a kernel that
// runs beside another one (the sweep beside the dense products, the verifier-row sweep beside
// the corrector) must leave room in its split for the other's CTAs. Everything not carved out
// is L1, which holds the sweep's loads in flight: the sweep is fastest with a small split.
constexpr int CARVEOUT_SMALL_KB = 64;    // sweep (2 KB a CTA), corrector, verification
constexpr int CARVEOUT_GEMM_KB = 132;    // a dense-product CTA (up to 97 KB) beside six sweep CTAs

// Sets the carveout preference of `func` on the current device once (kernels of the same
// signature are distinct entries: the registry is keyed by the function's address).
inline cudaError_t prefer_carveout_fn(const void* func, int kb) {
  static std::mutex mu;
  static std::vector<std::pair<const void*, int>> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (const auto& d : done)
    if (d.first == func && d.second == dev) return cudaSuccess;
  int max_smem = 0;
  e = cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  if (e != cudaSuccess) return e;
  int pct = max_smem > 0 ? (kb * 1024 * 100 + max_smem - 1) / max_smem : 100;
  if (pct > 100) pct = 100;
  e = cudaFuncSetAttribute(func, cudaFuncAttributePreferredSharedMemoryCarveout, pct);
  if (e == cudaSuccess) done.emplace_back(func, dev);
  return e;
}

template <typename Kernel>
inline cudaError_t prefer_carveout(Kernel kernel, int kb) {
  return prefer_carveout_fn(reinterpret_cast<const void*>(kernel), kb);
}

// ---------------------------------------------------------------- mbarriers and bulk copies
// Bounded waits: a wait gives up after a limit of SM cycles (wait_limit_cycles(), set by
// brisk_set_wait_limit and passed to kernels as an argument); the drain of copies still in
// flight after a give-up is bounded by the default limit.
constexpr long long DRAIN_LIMIT_CYCLES = 4000000000ll;  // about 2 s of SM clock
constexpr long long SHORT_WAIT_CYCLES = 1ll << 20;      // below this, waits poll without suspending
long long wait_limit_cycles();

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(su32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking test of the phase with the given parity (never suspends the thread).
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(su32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for a phase that is known to complete (the drain after a give-up), bounded by the
// default limit.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity) && clock64() - t0 < DRAIN_LIMIT_CYCLES) {
  }
}
// Orders this thread's earlier shared-memory accesses before later async-proxy (TMA, bulk copy)
// accesses of the same memory.
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// Launches `kernel` with the priority of `stream` as a launch attribute. Kernel nodes captured
// into a CUDA graph keep launch attributes, but not the priority of the stream they were captured
// from, so without it a replay of the tail's three-priority schedule runs every kernel at the
// default priority.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_prio(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                               cudaStream_t stream, Args&&... args) {
  int prio = 0;
  cudaError_t e = cudaStreamGetPriority(stream, &prio);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributePriority;
  attr[0].val.priority = prio;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

__device__ __forceinline__ void set_status(int32_t* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ float sigmoidf_(float x) { return 1.f / (1.f + expf(-x)); }

// ---------------------------------------------------------------- sweep
struct SweepSeg {
  const void* logits;     // [rows, V]
  int rows;               // rows in this segment
  int kout;               // entries to output per row (K for proposal rows, 1 for verifier rows)
  int32_t* out_ids;       // [rows, kout]
  float* out_logprob;     // [rows, kout] or nullptr
  float* out_lse;         // [rows]
  float* part_val;        // [rows, nchunk, KP]
  int32_t* part_id;       // [rows, nchunk, KP]
  float* part_m;          // [rows, nchunk]
  float* part_s;          // [rows, nchunk]
  int32_t* counters;      // [rows]
};

// Work layouts of the sweep: each warp its own (row, chunk), or each CTA one (row, split).
enum SweepMode { SWEEP_ROWS = 0, SWEEP_SPLIT = 1 };

struct SweepLaunch {
  SweepSeg seg[2];
  int nseg;
  int V;
  int mode;               // SweepMode
  int nchunk;             // chunks per row (a multiple of 4 for SWEEP_SPLIT)
  int KP;
  int dtype;              // brisk_dtype of the logits
  int32_t* status;
};

int sweep_chunks(int rows_per_tensor, int V, int dtype, int mode);
int kp_for(int K);
cudaError_t launch_sweep(const SweepLaunch& a, cudaStream_t stream);

// ---------------------------------------------------------------- dense products (SIMT, fp32 accumulate)
// C[m, n] = sum_k A(m, k) B(n, k), A(m,k) = A[m*lda + k], B(n,k) = transB ? B[k*ldb + n] : B[n*ldb + k].
cudaError_t gemm_simt(int M, int N, int K, const void* A, int a_dt, int lda, const void* B,
                      int b_dt, int ldb, bool transB, float* C, int ldc, cudaStream_t stream,
                      const float* bias = nullptr, int bias_period = 1);
// Tensor-core product on sm_103a: C = A B^T with A [M, K] and B [N, K] bf16 (row strides lda, ldb),
// fp32 accumulation; mode 0 stores fp32 C[m*ldc + n], mode 1 stores three bf16 parts whose sum
// is c to about 2^-24 relative (hi at [m*ldc + n], mid at [m*ldc + N + n], lo at [m*ldc + 2N + n]).
cudaError_t gemm_tc(int M, int N, int K, const void* A, int lda, const void* B, int ldb, int mode,
                    void* C, int ldc, int32_t* status, cudaStream_t stream);
// Up to two independent products of the same kind in one launch.
struct TcSpec {
  int M, N, K;
  const void* A;
  int lda;
  const void* B;
  int ldb;
  int mode;
  void* C;
  int ldc;
  const float* bias;   // optional fp32 [bias_period, N] added to row m as bias[m % bias_period] (mode 0)
  int bias_period;
  // Widest output tile (columns) to use, 0 for the default 256; narrower tiles give more CTAs
  // and a smaller pipeline stage. Read from the first product of a grouped launch.
  int max_bn;
};
// `stages` (2 or 4) sets the shared-memory pipeline depth: 2 leaves room on each SM for other
// kernels running concurrently.
// small_carveout: the kernel (a separate instantiation) prefers the small shared-memory
// carveout of the sweep, so that its CTAs can share SMs with sweep CTAs; the tiles must then fit
// it (64-wide, two stages: 49 KB).
cudaError_t gemm_tc_grouped(const TcSpec* spec, int nprob, int32_t* status, cudaStream_t stream,
                            int stages, bool small_carveout = false);
bool gemm_tc_supported(const void* A, int lda, const void* B, int ldb, int K);
// dst[i*ldd + j] = (dst type) src[i*lds + j], i < rows, j < cols (src[j*lds + i] with transpose).
cudaError_t copy2d(int rows, int cols, const void* src, int s_dt, int lds, void* dst, int d_dt,
                   int ldd, cudaStream_t stream, bool transpose = false);

// ---------------------------------------------------------------- corrector scan and verify
struct ScanArgs {
  int B, L, V, K, S, logits_dt;
  int select_mode, verify_mode;
  int do_select, do_verify;
  // corrector inputs
  const void* logits_q;
  const int32_t* cand_ids;
  const float* cand_logprob;
  const int32_t* x0;
  const float* u_sel;
  const float* G;        // [B*L, 2S] hidden shares of the GRU pre-activations (z | h)
  const float* posG;     // [L, 2S]   position shares of the GRU pre-activations (z | h)
  const float* G0;       // [B, S]    hidden-state part of Init
  const float* Tzh;      // [V, 2S]   token part of the GRU pre-activations (z | h)
  const float* U;        // [V, S]    residual rows: d = <s, U[c]>
  const float* T0;       // [V, S]    token part of Init

  const float* Fz;       // [S, 5]
  const float* Fh;       // [S, 5]
  const float* wg;       // [S + 5]
  float b_g, alpha;
  // same-state replay (App. B): feed the base selection forward instead of the head's, and
  // record its rank
  int base_prefix;
  int32_t* base_rank;    // [B, L] (base_prefix only)
  // select outputs (or verify inputs when do_select == 0)
  int32_t* sel_tokens;   // [B, L]
  float* refined;        // [B, L, K]
  // verify inputs / outputs
  const void* logits_p;
  const int32_t* argmax_p;  // [B, L]
  const float* lse_p;       // [B, L]
  const float* u_acc;
  const float* u_res;
  int32_t* accepted_len;
  int32_t* out_tokens;
  int32_t* correction;
  int32_t* next_anchor;
  int32_t* status;
};

// ---------------------------------------------------------------- distillation loss
struct DistillArgs {
  int B, L, V, K, logits_dt;
  const void* logits_p;        // [B, L, V] verifier logits
  const int32_t* cand_ids;     // [B, L, K]
  const float* cand_logprob;   // [B, L, K]
  const float* refined;        // [B, L, K]
  const int32_t* accepted_len; // [B]
  float beta;
  float* loss;                 // [1]
  float* grad;                 // [B, L, K] or nullptr
  float* partial;              // [B] per-sequence loss sums (workspace)
  int32_t* arrivals;           // zero on entry (workspace)
  int32_t* status;
};
cudaError_t launch_distill(const DistillArgs& a, cudaStream_t stream);

// ---------------------------------------------------------------- same-state replay
struct ReplayArgs {
  int B, L, V, K, logits_dt;
  const void* logits_p;        // [B, L, V]
  const float* lse_p;          // [B, L]
  const int32_t* cand_ids;     // [B, L, K]
  const float* cand_logprob;   // [B, L, K]
  const int32_t* base_rank;    // [B, L]
  const int32_t* head_tokens;  // [B, L]
  const float* u_acc;          // [B, L]
  int32_t* flags;              // [B, L]
  int32_t* first_breaker;      // [B]
  int32_t* status;
};
cudaError_t launch_replay(const ReplayArgs& a, cudaStream_t stream);

size_t scan_smem_bytes(int L, int K, int S, int V);
cudaError_t launch_scan(const ScanArgs& a, cudaStream_t stream);

// ---------------------------------------------------------------- contexts
// Unique id of the CUDA context current on this thread (cuCtxGetId; ids are never reused, so a
// device reset, which creates a new context, gives a new id). False when no context is current
// or the driver entry points are unavailable.
bool current_context_id(unsigned long long* id);

// ---------------------------------------------------------------- fused tail
// Serialises the use of the library's side streams: held while one call enqueues on them, and
// by graph creation from the start of its capture to the end.
std::mutex& side_stream_mutex();
// brisk_decode_tail with side_stream_mutex() already held by the caller.
brisk_status decode_tail_locked(const brisk_dims* d, const brisk_params* p, const void* tables,
                                const brisk_tail_io* io, int32_t select_mode, int32_t verify_mode,
                                void* ws, const brisk_events* ev, void* stream);

}  // namespace brisk
