// Tensor-core product C[m, n] = sum_k A[m, k] B[n, k] for bf16 A, B (both K-contiguous)
// with fp32 accumulation, on the 5th-generation tensor cores of sm_103a.
//
// One CTA computes one 128 x BN tile. A TMA producer thread streams 64-wide K
// slices of A and B into a 4-stage ring of 128-byte-swizzled shared-memory
// buffers; one thread issues tcgen05.mma (M = 128, N = BN, K = 16) into a TMEM
// accumulator and releases each stage with tcgen05.commit; then all four warps
// read their 32 TMEM lanes back with tcgen05.ld and write the tile. Every
// wait on an mbarrier is bounded (about 2 s of SM clock): on expiry the CTA records BRISK_ERR_TIMEOUT,
// drains what it started and frees its TMEM.
//
// Used for the corrector's one dense contraction (the MASK hidden states times
// the hidden projection, App. C.2 "64-dimensional projection of the MASK
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
constexpr long long WAIT_LIMIT_CYCLES = 4000000000ll;   // about 2 s of SM clock per wait

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
// Bounded wait for the phase with the given parity; false on expiry or abort. The SM cycle
// counter and the abort flag are only read every 64 polls.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (unsigned n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 63) == 0 && (*abort_flag || clock64() - t0 > WAIT_LIMIT_CYCLES)) return false;
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
  int ldc;
  int mtiles, ntiles;
  void* C;
  const float* bias;   // optional fp32 [bias_period, N], added to row m as bias[m % bias_period]
  int bias_period;
};

struct TcArgs {
  TcProblem p[2];   // one launch serves up to two independent products (grouped)
  int nprob;
  int tiles0;       // CTAs of problem 0
  int BN;           // tile columns (multiple of 16, <= 256), shared by both problems
  int tmem_cols;    // power of two >= max(32, BN)
  int32_t* status;
};

template <int TC_STAGES>
__global__ void __launch_bounds__(TC_THREADS, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmB0,
               const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
               const __grid_constant__ TcArgs a) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment of every stage buffer (required by the 128-byte swizzle atoms)
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int a_bytes = TC_BM * TC_BK * 2;
  const int b_bytes = a.BN * TC_BK * 2;
  uint8_t* sA = base;
  uint8_t* sB = base + TC_STAGES * a_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + TC_STAGES * b_bytes);
  uint64_t* empty = full + TC_STAGES;
  uint64_t* accum = empty + TC_STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pi = (a.nprob > 1 && (int)blockIdx.x >= a.tiles0) ? 1 : 0;
  const TcProblem& P = a.p[pi];
  const CUtensorMap* tmA = pi ? &tmA1 : &tmA0;
  const CUtensorMap* tmB = pi ? &tmB1 : &tmB0;
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
      if (kb >= TC_STAGES && !mbar_wait(&empty[s], ((kb / TC_STAGES) & 1) ^ 1, abort_flag)) {
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
      if (!mbar_wait(&full[s], (kb / TC_STAGES) & 1, abort_flag)) {
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
  // compete with TMA and the MMAs for the shared-memory pipe); the others wait at the barrier
  __syncthreads();
  if (threadIdx.x == 0) {
    const long long t0 = clock64();
    bool done = false;
    while (!(done = mbar_try_wait(accum, 0))) {
      if (*abort_flag || clock64() - t0 > WAIT_LIMIT_CYCLES) break;
      __nanosleep(128);
    }
    if (!done) *abort_flag = 1;
  }
  __syncthreads();
  tc_fence_after();
  // Every warp owns TMEM lanes [32*warp, 32*warp + 32) = tile rows: each thread holds one row
  // and writes it 32 columns at a time with 16-byte stores (a row segment per thread).
  if (!*abort_flag) {
    const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    const int row = m0 + warp * 32 + lane;
    const bool live = row < P.M;
    const float* brow = (P.bias && live) ? P.bias + (size_t)(row % P.bias_period) * P.N : nullptr;
    for (int c0 = 0; c0 < a.BN; c0 += 32) {
      float v[32];
      tmem_ld32(trow + c0, v);
      const int nb = n0 + c0;
      if (!live || nb >= P.N) continue;
      if (P.mode == 0) {
        float* Cr = static_cast<float*>(P.C) + (size_t)row * P.ldc + nb;
        if (brow) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (nb + 4 * q + 3 < P.N) {
              const float4 b = __ldg(reinterpret_cast<const float4*>(brow + nb) + q);
              v[4 * q] += b.x; v[4 * q + 1] += b.y; v[4 * q + 2] += b.z; v[4 * q + 3] += b.w;
            }
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (nb + 4 * q + 3 < P.N) {
            reinterpret_cast<float4*>(Cr)[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          } else {
            for (int e = 0; e < 4; ++e)
              if (nb + 4 * q + e < P.N) Cr[4 * q + e] = v[4 * q + e] + (brow ? brow[nb + 4 * q + e] : 0.f);
          }
        }
      } else {
        // three bf16 parts, hi + mid + lo = x to about 2^-24 relative
        __nv_bfloat16* Cr = static_cast<__nv_bfloat16*>(P.C) + (size_t)row * P.ldc + nb;
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
          if (nb + 8 * q + 7 < P.N) {
            reinterpret_cast<uint4*>(Cr)[q] = reinterpret_cast<const uint4*>(hi)[q];
            reinterpret_cast<uint4*>(Cr + P.N)[q] = reinterpret_cast<const uint4*>(mid)[q];
            reinterpret_cast<uint4*>(Cr + 2 * P.N)[q] = reinterpret_cast<const uint4*>(lo)[q];
          } else {
            for (int e = 0; e < 8; ++e)
              if (nb + 8 * q + e < P.N) {
                Cr[8 * q + e] = hi[8 * q + e];
                Cr[P.N + 8 * q + e] = mid[8 * q + e];
                Cr[2 * P.N + 8 * q + e] = lo[8 * q + e];
              }
          }
        }
      }
    }
  } else if (lane == 0) {
    set_status(a.status, BRISK_ERR_TIMEOUT);
    *abort_flag = 1;
  }
  // drain: the producer's loads complete on their own; wait (bounded) for the ones issued
  if (warp == 0 && lane == 0 && *abort_flag) {
    for (int kb = (issued > TC_STAGES ? issued - TC_STAGES : 0); kb < issued; ++kb) {
      const long long t0 = clock64();
      while (!mbar_try_wait(&full[kb % TC_STAGES], (kb / TC_STAGES) & 1) &&
             clock64() - t0 < WAIT_LIMIT_CYCLES) {
      }
    }
  }
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
                            int stages) {
  if (nprob < 1 || nprob > 2 || (stages != 2 && stages != 4)) return cudaErrorInvalidValue;
  int nmax = 0;
  for (int i = 0; i < nprob; ++i) nmax = spec[i].N > nmax ? spec[i].N : nmax;
  int BN = ((nmax + 15) / 16) * 16;
  if (BN > 256) BN = 256;
  int cols = 32;
  while (cols < BN) cols *= 2;
  CUtensorMap maps[4];
  TcArgs a{};
  a.nprob = nprob;
  a.BN = BN;
  a.tmem_cols = cols;
  a.status = status;
  int total = 0;
  for (int i = 0; i < 2; ++i) {
    const TcSpec& q = spec[i < nprob ? i : 0];
    if (!make_map(&maps[2 * i], q.A, q.M, q.K, q.lda, TC_BM) ||
        !make_map(&maps[2 * i + 1], q.B, q.N, q.K, q.ldb, BN))
      return cudaErrorInvalidValue;
    if (i >= nprob) continue;
    TcProblem& P = a.p[i];
    P.M = q.M; P.N = q.N; P.K = q.K; P.mode = q.mode; P.ldc = q.ldc; P.C = q.C;
    P.bias = q.bias;
    P.bias_period = q.bias_period > 0 ? q.bias_period : 1;
    P.mtiles = (q.M + TC_BM - 1) / TC_BM;
    P.ntiles = (q.N + BN - 1) / BN;
    if (i == 0) a.tiles0 = P.mtiles * P.ntiles;
    total += P.mtiles * P.ntiles;
  }
  if (total == 0) return cudaSuccess;
  const size_t smem = gemm_tc_smem(BN, stages);
  if (stages == 2) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e == cudaSuccess) e = prefer_carveout(gemm_tc_kernel<2>, CARVEOUT_GEMM_KB);
    if (e != cudaSuccess) return e;
    gemm_tc_kernel<2><<<total, TC_THREADS, smem, stream>>>(maps[0], maps[1], maps[2], maps[3], a);
  } else {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e == cudaSuccess) e = prefer_carveout(gemm_tc_kernel<4>, CARVEOUT_GEMM_KB);
    if (e != cudaSuccess) return e;
    gemm_tc_kernel<4><<<total, TC_THREADS, smem, stream>>>(maps[0], maps[1], maps[2], maps[3], a);
  }
  return cudaGetLastError();
}

cudaError_t gemm_tc(int M, int N, int K, const void* A, int lda, const void* B, int ldb, int mode,
                    void* C, int ldc, int32_t* status, cudaStream_t stream) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  const TcSpec s{M, N, K, A, lda, B, ldb, mode, C, ldc, nullptr, 0};
  return gemm_tc_grouped(&s, 1, status, stream, 4);
}

}  // namespace brisk
