// Tensor-core product C[m, n] = sum_k A[m, k] B[n, k] for bf16 A, B (both K-contiguous)
// with fp32 accumulation, on the 5th-generation tensor cores of sm_103a.
//
// One CTA computes one 128 x BN tile. A TMA producer thread streams 64-wide K slices of A and
// B into a ring of 128-byte-swizzled shared-memory buffers; one thread issues tcgen05.mma
// (M = 128, N = BN, K = 16) into a TMEM accumulator and releases each stage with
// tcgen05.commit. The epilogue reads TMEM 32 columns at a time (tcgen05.ld), stages each chunk
// in one of several shared-memory buffers (the ring is free by then) and writes it with a TMA
// tensor store, so that staging the next chunks overlaps the stores in flight. Every wait on
// an mbarrier is bounded (a kernel argument, by default about 2 s of SM clock): on expiry the
// CTA records BRISK_ERR_TIMEOUT, drains what it started (its TMA loads and the tensor-core
// operations it issued, each drain wait bounded by the default limit) and frees its TMEM.
//
// Used for the corrector's one dense contraction (the MASK hidden states times
// the hidden projection, App. C.3 "64-dimensional projection of the MASK
// hidden state") and for the products that follow it, where an fp32 operand
// enters as the sum of three bf16 parts (hi + mid + lo) so that bf16 tensor
// cores keep fp32-level accuracy.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "brisk_internal.cuh"

namespace brisk {

namespace {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;               // one 128-byte swizzle row of bf16
constexpr int TC_STAGES_MAX = 4;
constexpr int TC_THREADS = 128;

// Bounded wait for the phase with the given parity; false on expiry (more than `limit` SM
// cycles) or abort. With a long limit the thread may suspend in try_wait and the cycle counter
// and the abort flag are read every 64 polls; a short limit (tests of the failure path) polls
// with test_wait and reads the counter every poll, so that it expires after `limit` cycles.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          long long limit) {
  if (limit < SHORT_WAIT_CYCLES) {
    const long long t0 = clock64();
    for (;;) {
      if (mbar_test(bar, parity)) return true;
      if (*abort_flag || clock64() - t0 > limit) return false;
    }
  }
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (unsigned n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 63) == 0 && (*abort_flag || clock64() - t0 > limit)) return false;
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(su32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(su32(bar)), "r"(x), "r"(y)
      : "memory");
}
// TMA tensor store of a box staged in shared memory (bulk-group completion).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(su32(src)), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until at most n (0, 1 or 3) committed bulk groups still read shared memory.
__device__ __forceinline__ void bulk_wait_read(int n) {
  if (n >= 3) asm volatile("cp.async.bulk.wait_group.read 3;" ::: "memory");
  else if (n == 1) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
  else asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D(tmem) (+)= A(smem desc) * B(smem desc)^T, kind::f16 (bf16 inputs), fp32 accumulator.
__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                     uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
      : "memory");
}
// 32 lanes x 32 consecutive fp32 columns of TMEM, waited for before returning.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

// Shared-memory matrix descriptor of a K-major tile stored as 8-row x 128-byte
// swizzle atoms (the layout TMA writes with 128-byte swizzling): start address,
// leading offset 16 B (unused by this layout), 1024 B between 8-row groups,
// descriptor version 1, swizzle mode 128 B.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(16 >> 4) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

struct TcProblem {
  int M, N, K;
  int mode;         // 0: fp32 C[m*ldc + n]; 1: bf16 parts hi, mid, lo at [m*ldc + {0, N, 2N} + n]
  int mtiles, ntiles;
  const float* bias;   // optional fp32 [bias_period, N], added to row m as bias[m % bias_period]
  int bias_period;
};

// Tensor maps of one launch: A and B of each problem, and the output boxes (mode 0: one fp32
// map [M, N]; mode 1: one bf16 map [M, N] per part).
struct TcMaps {
  CUtensorMap a[2], b[2], c[2][3];
};

struct TcArgs {
  TcProblem p[2];   // one launch serves up to two independent products (grouped)
  int nprob;
  int tiles0;       // CTAs of problem 0
  int BN;           // tile columns (multiple of 16, <= 256), shared by both problems
  int tmem_cols;    // power of two >= max(32, BN)
  long long wait_limit;   // SM cycles a pipeline or accumulator wait spins before it gives up
  int32_t* status;
};

// Staging of one 32-column output chunk: fp32 (mode 0) or three bf16 parts (mode 1).
constexpr int TC_OUT_CHUNK_F32 = TC_BM * 32 * 4;
constexpr int TC_OUT_CHUNK_BF16X3 = 3 * TC_BM * 32 * 2;

// SMALL_CARVEOUT does not change the code: it makes a separate kernel whose shared-memory
// carveout preference (a per-kernel attribute) is the sweep's.
template <int TC_STAGES, bool SMALL_CARVEOUT = false>
__global__ void __launch_bounds__(TC_THREADS, 1)
gemm_tc_kernel(const __grid_constant__ TcMaps maps, const __grid_constant__ TcArgs a) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment of every stage buffer (required by the 128-byte swizzle atoms)
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int a_bytes = TC_BM * TC_BK * 2;
  const int b_bytes = a.BN * TC_BK * 2;
  uint8_t* sA = base;
  uint8_t* sB = base + TC_STAGES * a_bytes;
  const int ring = TC_STAGES * (a_bytes + b_bytes);   // reused by the epilogue's output stages
  uint64_t* full = reinterpret_cast<uint64_t*>(base + ring);
  uint64_t* empty = full + TC_STAGES;
  uint64_t* accum = empty + TC_STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pi = (a.nprob > 1 && (int)blockIdx.x >= a.tiles0) ? 1 : 0;
  const TcProblem& P = a.p[pi];
  const CUtensorMap* tmA = &maps.a[pi];
  const CUtensorMap* tmB = &maps.b[pi];
  const int tile = (int)blockIdx.x - (pi ? a.tiles0 : 0);
  const int m0 = (tile % P.mtiles) * TC_BM, n0 = (tile / P.mtiles) * a.BN;
  const int nk = (P.K + TC_BK - 1) / TC_BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < TC_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) tmem_alloc(tmem_slot, a.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  int issued = 0;    // stages the producer started (for draining on abort)
  if (warp == 0 && lane == 0) {
    // TMA producer
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % TC_STAGES;
      if (kb >= TC_STAGES &&
          !mbar_wait(&empty[s], ((kb / TC_STAGES) & 1) ^ 1, abort_flag, a.wait_limit)) {
        *abort_flag = 1;
        break;
      }
      mbar_expect_tx(&full[s], a_bytes + b_bytes);
      tma_load_2d(sA + s * a_bytes, tmA, &full[s], kb * TC_BK, m0);
      tma_load_2d(sB + s * b_bytes, tmB, &full[s], kb * TC_BK, n0);
      issued = kb + 1;
    }
  } else if (warp == 1 && lane == 0) {
    // MMA issuer
    const uint32_t idesc = idesc_bf16(TC_BM, a.BN);
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % TC_STAGES;
      if (!mbar_wait(&full[s], (kb / TC_STAGES) & 1, abort_flag, a.wait_limit)) {
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint64_t ad = sw128_desc(su32(sA + s * a_bytes));
      const uint64_t bd = sw128_desc(su32(sB + s * b_bytes));
#pragma unroll
      for (int kk = 0; kk < TC_BK / 16; ++kk)   // 16 bf16 = 32 bytes per step: +2 in 16-byte units
        umma(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
      umma_commit(&empty[s]);
    }
    umma_commit(accum);
  }
  // epilogue: one thread waits for the accumulator (with back-off, so that polling does not
  // compete with TMA and the MMAs for the shared-memory pipe); the others wait at the barrier.
  // The MMA thread has issued its commit to `accum` before this barrier, aborted or not.
  __syncthreads();
  if (threadIdx.x == 0) {
    const long long t0 = clock64();
    bool done = false;
    while (!(done = mbar_test(accum, 0))) {
      if (*abort_flag || clock64() - t0 > a.wait_limit) break;
      if (a.wait_limit >= SHORT_WAIT_CYCLES) __nanosleep(128);
    }
    if (!done) {
      *abort_flag = 1;
      // the tensor-core operations already issued still write TMEM and read the ring: the
      // commit covers all of them, so wait for it before TMEM is freed
      mbar_drain(accum, 0);
    }
  }
  // drain: the producer's loads complete on their own; wait (bounded) for the ones issued
  if (warp == 0 && lane == 0 && *abort_flag) {
    for (int kb = (issued > TC_STAGES ? issued - TC_STAGES : 0); kb < issued; ++kb)
      mbar_drain(&full[kb % TC_STAGES], (kb / TC_STAGES) & 1);
  }
  __syncthreads();
  tc_fence_after();
  const bool ok = !*abort_flag;
  if (!ok && threadIdx.x == 0) set_status(a.status, BRISK_ERR_TIMEOUT);

  // Epilogue. Warp w holds tile rows [32w, 32w + 32) in its TMEM lanes, one row a thread. A
  // finished 32-column chunk is staged in shared memory and written by TMA tensor stores
  // (which clip rows and columns outside the product); chunk c uses stage buffer c % nbuf, so
  // up to nbuf stores are in flight while the next chunks are staged.
  if (ok) {
    const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    const int rt = warp * 32 + lane;                 // row within the tile
    const int row = m0 + rt;
    const float* brow = (P.bias && row < P.M) ? P.bias + (size_t)(row % P.bias_period) * P.N : nullptr;
    const int chunk_bytes = P.mode == 0 ? TC_OUT_CHUNK_F32 : TC_OUT_CHUNK_BF16X3;
    const int fit = ring / chunk_bytes;
    const int nbuf = fit >= 4 ? 4 : (fit >= 2 ? 2 : 1);
    for (int c = 0, ci = 0; c < a.BN; c += 32, ++ci) {
      float v[32];
      tmem_ld32(trow + c, v);
      const int nb = n0 + c;
      if (brow) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (nb + 4 * q + 3 < P.N) {
            const float4 b = __ldg(reinterpret_cast<const float4*>(brow + nb) + q);
            v[4 * q] += b.x; v[4 * q + 1] += b.y; v[4 * q + 2] += b.z; v[4 * q + 3] += b.w;
          } else {
            for (int e = 0; e < 4; ++e)
              if (nb + 4 * q + e < P.N) v[4 * q + e] += brow[nb + 4 * q + e];
          }
      }
      uint8_t* stage = base + (ci % nbuf) * chunk_bytes;
      if (threadIdx.x == 0) bulk_wait_read(nbuf - 1);   // the store that last used `stage` has read it
      __syncthreads();
      if (P.mode == 0) {
        float4* st = reinterpret_cast<float4*>(stage + rt * 128);
#pragma unroll
        for (int q = 0; q < 8; ++q) st[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      } else {
        // three bf16 parts, hi + mid + lo = x to about 2^-24 relative
        __align__(16) __nv_bfloat16 hi[32], mid[32], lo[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          hi[j] = __float2bfloat16_rn(v[j]);
          const float r1 = v[j] - __bfloat162float(hi[j]);
          mid[j] = __float2bfloat16_rn(r1);
          lo[j] = __float2bfloat16_rn(r1 - __bfloat162float(mid[j]));
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          reinterpret_cast<uint4*>(stage + rt * 64)[q] = reinterpret_cast<const uint4*>(hi)[q];
          reinterpret_cast<uint4*>(stage + TC_BM * 64 + rt * 64)[q] = reinterpret_cast<const uint4*>(mid)[q];
          reinterpret_cast<uint4*>(stage + 2 * TC_BM * 64 + rt * 64)[q] = reinterpret_cast<const uint4*>(lo)[q];
        }
      }
      fence_async_smem();
      __syncthreads();
      if (threadIdx.x == 0) {
        if (P.mode == 0) {
          tma_store_2d(&maps.c[pi][0], stage, nb, m0);
        } else {
#pragma unroll
          for (int part = 0; part < 3; ++part)
            tma_store_2d(&maps.c[pi][part], stage + part * TC_BM * 64, nb, m0);
        }
        bulk_commit();
      }
    }
  }
  if (threadIdx.x == 0) bulk_wait0();             // stores complete before the CTA ends
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, a.tmem_cols);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor [rows, cols] with row stride ld (elements), boxes of 64 x box_rows, 128-byte swizzle.
bool make_map(CUtensorMap* map, const void* ptr, int rows, int cols, int ld, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(TC_BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output map: [rows, cols] of fp32 or bf16 with row stride ld (elements), boxes of 32 x 128, no
// swizzle (the epilogue stages a chunk row-major).
bool make_out_map(CUtensorMap* map, const void* ptr, bool f32, int rows, int cols, int ld) {
  auto fn = encode_fn();
  if (!fn) return false;
  const int es = f32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(ptr) % 16 != 0 || ((size_t)ld * es) % 16 != 0) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * es};
  cuuint32_t box[2] = {32, static_cast<cuuint32_t>(TC_BM)};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
            const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

std::atomic<long long> g_wait_limit{DRAIN_LIMIT_CYCLES};

}  // namespace

long long wait_limit_cycles() { return g_wait_limit.load(std::memory_order_relaxed); }

namespace {

int tc_bn(int nmax) {
  int BN = ((nmax + 15) / 16) * 16;
  return BN > 256 ? 256 : BN;
}

}  // namespace

size_t gemm_tc_smem(int BN, int stages) {
  return 1024 + stages * (TC_BM * TC_BK * 2 + BN * TC_BK * 2) + (2 * TC_STAGES_MAX + 1) * 8 + 16;
}

bool gemm_tc_supported(const void* A, int lda, const void* B, int ldb, int K) {
  return encode_fn() != nullptr && (reinterpret_cast<uintptr_t>(A) % 16 == 0) &&
         (reinterpret_cast<uintptr_t>(B) % 16 == 0) && (lda % 8 == 0) && (ldb % 8 == 0) && K >= 1;
}

// One or two products C = A B^T, A [M, K] (row stride lda) and B [N, K] (row stride ldb) bf16,
// fp32 accumulation, in one launch.
cudaError_t gemm_tc_grouped(const TcSpec* spec, int nprob, int32_t* status, cudaStream_t stream,
                            int stages, bool small_carveout) {
  if (nprob < 1 || nprob > 2 || (stages != 2 && stages != 4)) return cudaErrorInvalidValue;
  if (small_carveout && stages != 2) return cudaErrorInvalidValue;
  int nmax = 0;
  for (int i = 0; i < nprob; ++i) nmax = spec[i].N > nmax ? spec[i].N : nmax;
  if (spec[0].max_bn >= 16 && nmax > spec[0].max_bn) nmax = spec[0].max_bn;
  const int BN = tc_bn(nmax);
  int cols = 32;
  while (cols < BN) cols *= 2;
  TcMaps maps;
  TcArgs a{};
  a.nprob = nprob;
  a.BN = BN;
  a.tmem_cols = cols;
  a.wait_limit = wait_limit_cycles();
  a.status = status;
  int total = 0;
  for (int i = 0; i < 2; ++i) {
    const TcSpec& q = spec[i < nprob ? i : 0];
    if (!make_map(&maps.a[i], q.A, q.M, q.K, q.lda, TC_BM) ||
        !make_map(&maps.b[i], q.B, q.N, q.K, q.ldb, BN))
      return cudaErrorInvalidValue;
    if (q.mode == 0) {
      if (!make_out_map(&maps.c[i][0], q.C, true, q.M, q.N, q.ldc)) return cudaErrorInvalidValue;
      maps.c[i][1] = maps.c[i][2] = maps.c[i][0];
    } else {
      for (int part = 0; part < 3; ++part)
        if (!make_out_map(&maps.c[i][part], static_cast<const __nv_bfloat16*>(q.C) + (size_t)part * q.N,
                          false, q.M, q.N, q.ldc))
          return cudaErrorInvalidValue;
    }
    if (i >= nprob) continue;
    TcProblem& P = a.p[i];
    P.M = q.M; P.N = q.N; P.K = q.K; P.mode = q.mode;
    P.bias = q.bias;
    P.bias_period = q.bias_period > 0 ? q.bias_period : 1;
    P.mtiles = (q.M + TC_BM - 1) / TC_BM;
    P.ntiles = (q.N + BN - 1) / BN;
    if (i == 0) a.tiles0 = P.mtiles * P.ntiles;
    total += P.mtiles * P.ntiles;
  }
  if (total == 0) return cudaSuccess;
  const size_t smem = gemm_tc_smem(BN, stages);
  if (small_carveout && smem > (size_t)(CARVEOUT_SMALL_KB - 1) * 1024) return cudaErrorInvalidValue;
  auto kernel = small_carveout ? gemm_tc_kernel<2, true>
                               : (stages == 2 ? gemm_tc_kernel<2> : gemm_tc_kernel<4>);
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e == cudaSuccess) e = prefer_carveout(kernel, small_carveout ? CARVEOUT_SMALL_KB : CARVEOUT_GEMM_KB);
  if (e != cudaSuccess) return e;
  e = launch_prio(kernel, dim3(total), dim3(TC_THREADS), smem, stream, maps, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t gemm_tc(int M, int N, int K, const void* A, int lda, const void* B, int ldb, int mode,
                    void* C, int ldc, int32_t* status, cudaStream_t stream) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  const TcSpec s{M, N, K, A, lda, B, ldb, mode, C, ldc, nullptr, 0, 0};
  return gemm_tc_grouped(&s, 1, status, stream, 4);
}

}  // namespace brisk

extern "C" int64_t brisk_set_wait_limit(int64_t cycles) {
  const long long v = cycles > 0 ? (long long)cycles : brisk::DRAIN_LIMIT_CYCLES;
  return (int64_t)brisk::g_wait_limit.exchange(v);
}
