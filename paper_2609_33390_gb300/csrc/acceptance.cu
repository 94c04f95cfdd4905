// Acceptance profile and risk-reward position weights (Sec. 2.2; Sec. 3.2 Eqs. 2-3).
//
// brisk_acceptance_counts: a per-step histogram of how far verification reached, as running
// per-position counts (device, integer atomics: the sums do not depend on timing).
// brisk_acceptance_weights / brisk_tpf_isd: the closed forms of the length law, TPF, FPT and
// the weights' derivative, on the host in double precision (M <= 64 positions).
#include <math.h>

#include "brisk_internal.cuh"

namespace brisk {
namespace {

constexpr int ACC_THREADS = 256;

// One CTA counts, in shared memory, the blocks of its stride that reached and accepted each
// position, then adds them to the global counts.
__global__ void __launch_bounds__(ACC_THREADS)
acceptance_counts_kernel(const int32_t* __restrict__ accepted_len, int B, int L,
                         unsigned long long* __restrict__ counts) {
  __shared__ unsigned int reach[64], accept[64];
  for (int i = threadIdx.x; i < L; i += ACC_THREADS) reach[i] = accept[i] = 0u;
  __syncthreads();
  for (int b = blockIdx.x * ACC_THREADS + threadIdx.x; b < B; b += gridDim.x * ACC_THREADS) {
    int len = accepted_len[b];
    len = len < 0 ? 0 : (len > L ? L : len);
    // reached positions 0..len (position len is reached unless len == L), accepted 0..len-1
    for (int i = 0; i < L; ++i) {
      if (i <= len) atomicAdd(&reach[i], 1u);
      if (i < len) atomicAdd(&accept[i], 1u);
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < L; i += ACC_THREADS) {
    if (reach[i]) atomicAdd(&counts[i], (unsigned long long)reach[i]);
    if (accept[i]) atomicAdd(&counts[L + i], (unsigned long long)accept[i]);
  }
}

}  // namespace
}  // namespace brisk

using namespace brisk;

extern "C" brisk_status brisk_acceptance_counts(const int32_t* accepted_len, int32_t B, int32_t L,
                                                unsigned long long* counts, void* stream) {
  if (L < 1 || L > 64 || B < 0 || !counts || (B > 0 && !accepted_len)) return BRISK_ERR_INVALID_ARG;
  if (B == 0) return BRISK_OK;
  const int grid = (B + ACC_THREADS - 1) / ACC_THREADS < 64 ? (B + ACC_THREADS - 1) / ACC_THREADS : 64;
  acceptance_counts_kernel<<<grid, ACC_THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
      accepted_len, B, L, counts);
  return cudaGetLastError() == cudaSuccess ? BRISK_OK : BRISK_ERR_CUDA;
}

extern "C" double brisk_tpf_isd(int32_t N, double r) {
  if (N < 2 || !(r >= 0.0 && r <= 1.0)) return NAN;
  const double q = 1.0 - r;
  double num = 2.0, qi = 1.0;
  for (int i = 1; i <= N - 2; ++i) {
    qi *= q;
    num += qi;
  }
  return num / (2.0 - qi * q);   // qi * q = q^(N-1)
}

extern "C" brisk_status brisk_isd_costs(int32_t M, double* g, double* c) {
  if (M < 1 || M > 64 || !g || !c) return BRISK_ERR_INVALID_ARG;
  for (int k = 0; k <= M; ++k) {
    g[k] = 2.0 + (k < M - 1 ? k : M - 1);
    c[k] = k < M ? 2.0 : 1.0;
  }
  return BRISK_OK;
}

extern "C" brisk_status brisk_acceptance_weights(int32_t M, const double* a, const double* g,
                                                 const double* c, double eps, double* tpf,
                                                 double* w_raw, double* w_bar) {
  if (M < 1 || M > 64 || !a) return BRISK_ERR_INVALID_ARG;
  for (int i = 0; i < M; ++i)
    if (!(a[i] >= 0.0 && a[i] <= 1.0)) return BRISK_ERR_INVALID_ARG;
  auto gk = [&](int k) { return g ? g[k] : (double)(k + 1); };
  auto ck = [&](int k) { return c ? c[k] : 1.0; };
  // prefix[k] = a_0 ... a_{k-1}, suffix products let dA_k/da_i skip a_i without dividing
  double prefix[65];
  prefix[0] = 1.0;
  for (int k = 1; k <= M; ++k) prefix[k] = prefix[k - 1] * a[k - 1];
  double G = 0.0, C = 0.0;
  for (int k = 0; k <= M; ++k) {
    const double pr = k < M ? prefix[k] * (1.0 - a[k]) : prefix[M];
    G += pr * gk(k);
    C += pr * ck(k);
  }
  if (!(G != 0.0) || !(C != 0.0)) return BRISK_ERR_INVALID_ARG;
  if (tpf) *tpf = G / C;
  if (!w_raw && !w_bar) return BRISK_OK;
  double w[64], wsum = 0.0;
  for (int i = 0; i < M; ++i) {
    // dPr(L=k)/da_i: k > i through A_k (the product without a_i), k == i through (1 - a_i)
    double dG = 0.0, dC = 0.0;
    double without_i = prefix[i];   // a_0 ... a_{i-1}, then times a_{i+1} ... a_{k-1}
    for (int k = i + 1; k <= M; ++k) {
      if (k > i + 1) without_i *= a[k - 1];
      const double d = k < M ? without_i * (1.0 - a[k]) : without_i;
      dG += d * gk(k);
      dC += d * ck(k);
    }
    dG -= prefix[i] * gk(i);
    dC -= prefix[i] * ck(i);
    // FPT = C / G
    const double dfpt = (dC * G - C * dG) / (G * G);
    w[i] = -dfpt * a[i] * (1.0 - a[i]);
    wsum += w[i];
  }
  for (int i = 0; i < M; ++i) {
    if (w_raw) w_raw[i] = w[i];
    if (w_bar) w_bar[i] = M * w[i] / (wsum + eps);
  }
  return BRISK_OK;
}
