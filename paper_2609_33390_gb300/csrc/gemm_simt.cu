// Plain tiled fp32 dense products and a conversion copy. They serve the one-off
// folding of the frozen vocabulary rows into the corrector tables
// (App. C.3: E, E_out and the backbone are frozen at inference) and the fp32
// configurations; every product accumulates in fp32.
#include "brisk_internal.cuh"

namespace brisk {

namespace {

constexpr int TM = 64, TN = 64, TK = 16;

template <typename TA, typename TB>
__global__ void __launch_bounds__(256)
gemm_simt_kernel(int M, int N, int K, const TA* __restrict__ A, int lda,
                 const TB* __restrict__ B, int ldb, int transB, float* __restrict__ C, int ldc,
                 const float* __restrict__ bias, int bias_period) {
  __shared__ float As[TK][TM + 4];
  __shared__ float Bs[TK][TN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const long long m0 = (long long)blockIdx.y * TM, n0 = (long long)blockIdx.x * TN;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int e = threadIdx.x; e < TM * TK; e += 256) {
      const int mm = e / TK, kk = e % TK;
      const long long gm = m0 + mm;
      const int gk = k0 + kk;
      As[kk][mm] = (gm < M && gk < K) ? to_f32(A[gm * lda + gk]) : 0.f;
    }
    for (int e = threadIdx.x; e < TN * TK; e += 256) {
      int nn, kk;
      if (transB) { kk = e / TN; nn = e % TN; } else { nn = e / TK; kk = e % TK; }
      const long long gn = n0 + nn;
      const int gk = k0 + kk;
      float v = 0.f;
      if (gn < N && gk < K) v = to_f32(transB ? B[(long long)gk * ldb + gn] : B[gn * ldb + gk]);
      Bs[kk][nn] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const long long gm = m0 + ty * 4 + i;
    if (gm >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const long long gn = n0 + tx * 4 + j;
      if (gn < N) C[gm * ldc + gn] = acc[i][j] + (bias ? bias[(gm % bias_period) * N + gn] : 0.f);
    }
  }
}

// Products with few rows (M <= SKINNY_MAX_M, B not transposed): a warp per output column n,
// lane l accumulating k = l, l + 32, ... for every row, then one warp sum per row. One pass over
// k with all loads in flight, where the tiled kernel would run a k-loop of K / 16 dependent
// steps on a single CTA (an 8 x 64 product over k = 512: about 65 us in it, a few us here).
constexpr int SKINNY_MAX_M = 16;
constexpr int SKINNY_WARPS = 8;

template <typename TA, typename TB>
__global__ void __launch_bounds__(SKINNY_WARPS * 32)
gemm_skinny_kernel(int M, int N, int K, const TA* __restrict__ A, int lda,
                   const TB* __restrict__ B, int ldb, float* __restrict__ C, int ldc,
                   const float* __restrict__ bias, int bias_period) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long n = (long long)blockIdx.x * SKINNY_WARPS + warp;
  if (n >= N) return;
  float acc[SKINNY_MAX_M];
#pragma unroll
  for (int m = 0; m < SKINNY_MAX_M; ++m) acc[m] = 0.f;
  const TB* brow = B + n * ldb;
  for (int k = lane; k < K; k += 32) {
    const float b = to_f32(brow[k]);
#pragma unroll
    for (int m = 0; m < SKINNY_MAX_M; ++m)
      if (m < M) acc[m] = fmaf(to_f32(A[(long long)m * lda + k]), b, acc[m]);
  }
#pragma unroll
  for (int m = 0; m < SKINNY_MAX_M; ++m) {
    if (m >= M) break;
    const float v = warp_sum(acc[m]);
    if (lane == 0) C[(long long)m * ldc + n] = v + (bias ? bias[(m % bias_period) * N + n] : 0.f);
  }
}

template <typename TS, typename TD>
__global__ void copy2d_kernel(int rows, int cols, const TS* __restrict__ src, int lds,
                              TD* __restrict__ dst, int ldd, int transpose) {
  const long long n = (long long)rows * cols;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n;
       e += (long long)gridDim.x * blockDim.x) {
    const long long i = e / cols, j = e % cols;
    const float v = to_f32(transpose ? src[j * lds + i] : src[i * lds + j]);
    if constexpr (sizeof(TD) == 4) dst[i * ldd + j] = v;
    else dst[i * ldd + j] = __float2bfloat16_rn(v);
  }
}

template <typename TA, typename TB>
cudaError_t gemm_t(int M, int N, int K, const void* A, int lda, const void* B, int ldb,
                   bool transB, float* C, int ldc, cudaStream_t stream, const float* bias,
                   int bias_period) {
  if (M <= SKINNY_MAX_M && !transB) {
    const unsigned grid = (unsigned)((N + SKINNY_WARPS - 1) / SKINNY_WARPS);
    const cudaError_t e = launch_prio(
        gemm_skinny_kernel<TA, TB>, dim3(grid), dim3(SKINNY_WARPS * 32), 0, stream, M, N, K,
        static_cast<const TA*>(A), lda, static_cast<const TB*>(B), ldb, C, ldc, bias,
        bias_period > 0 ? bias_period : 1);
    return e != cudaSuccess ? e : cudaGetLastError();
  }
  const dim3 grid((N + TN - 1) / TN, (M + TM - 1) / TM);
  const cudaError_t e = launch_prio(gemm_simt_kernel<TA, TB>, grid, dim3(256), 0, stream,
      M, N, K, static_cast<const TA*>(A), lda, static_cast<const TB*>(B), ldb, transB ? 1 : 0, C, ldc,
      bias, bias_period > 0 ? bias_period : 1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <typename TS>
cudaError_t copy_t(int rows, int cols, const void* src, int lds, void* dst, int d_dt, int ldd,
                   bool transpose, cudaStream_t stream) {
  const long long n = (long long)rows * cols;
  const unsigned grid = (unsigned)((n + 255) / 256 > 4096 ? 4096 : (n + 255) / 256);
  if (d_dt == BRISK_DT_F32)
    copy2d_kernel<TS, float><<<grid, 256, 0, stream>>>(rows, cols, static_cast<const TS*>(src), lds,
                                                       static_cast<float*>(dst), ldd, transpose);
  else
    copy2d_kernel<TS, __nv_bfloat16><<<grid, 256, 0, stream>>>(
        rows, cols, static_cast<const TS*>(src), lds, static_cast<__nv_bfloat16*>(dst), ldd,
        transpose);
  return cudaGetLastError();
}

}  // namespace

cudaError_t gemm_simt(int M, int N, int K, const void* A, int a_dt, int lda, const void* B,
                      int b_dt, int ldb, bool transB, float* C, int ldc, cudaStream_t stream,
                      const float* bias, int bias_period) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  if (a_dt == BRISK_DT_BF16 && b_dt == BRISK_DT_BF16)
    return gemm_t<__nv_bfloat16, __nv_bfloat16>(M, N, K, A, lda, B, ldb, transB, C, ldc, stream,
                                                 bias, bias_period);
  if (a_dt == BRISK_DT_F32 && b_dt == BRISK_DT_BF16)
    return gemm_t<float, __nv_bfloat16>(M, N, K, A, lda, B, ldb, transB, C, ldc, stream, bias,
                                        bias_period);
  if (a_dt == BRISK_DT_BF16 && b_dt == BRISK_DT_F32)
    return gemm_t<__nv_bfloat16, float>(M, N, K, A, lda, B, ldb, transB, C, ldc, stream, bias,
                                        bias_period);
  return gemm_t<float, float>(M, N, K, A, lda, B, ldb, transB, C, ldc, stream, bias, bias_period);
}

cudaError_t copy2d(int rows, int cols, const void* src, int s_dt, int lds, void* dst, int d_dt,
                   int ldd, cudaStream_t stream, bool transpose) {
  if (rows <= 0 || cols <= 0) return cudaSuccess;
  if (s_dt == BRISK_DT_BF16)
    return copy_t<__nv_bfloat16>(rows, cols, src, lds, dst, d_dt, ldd, transpose, stream);
  return copy_t<float>(rows, cols, src, lds, dst, d_dt, ldd, transpose, stream);
}

}  // namespace brisk
