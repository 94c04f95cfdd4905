// Same-state replay diagnostics (App. B, "Same-state replay", Eq. 6): with the factual base
// prefix, the base q_i (normalised over the full vocabulary), the verifier p_i and one draw u_i
// fixed, compare the base token and the head's token at every position under
// alpha_i(x) = min(1, p_i(x) / q_i(x)), J_i(x) = [u_i < alpha_i(x)].
//
// One warp per sequence, lane l holding positions l and l + 32. The first breaker (the first
// position whose base token the draw rejects) comes from a ballot; rescues are counted there
// and regressions before it.
#include "brisk_internal.cuh"

namespace brisk {
namespace {

constexpr int REPLAY_WARPS = 4;

__device__ __forceinline__ float logit_at(const void* base, int dt, size_t idx) {
  if (dt == BRISK_DT_BF16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(base)[idx]);
  return reinterpret_cast<const float*>(base)[idx];
}

__global__ void __launch_bounds__(REPLAY_WARPS * 32)
replay_kernel(const __grid_constant__ ReplayArgs a) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * REPLAY_WARPS + (threadIdx.x >> 5);
  if (b >= a.B) return;
  const int L = a.L, K = a.K;
  bool jb[2] = {true, true}, jh[2] = {true, true}, changed[2] = {false, false};
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    if (i >= L) continue;
    const size_t row = (size_t)b * L + i;
    int rb = a.base_rank[row];
    if (rb < 0 || rb >= K) { set_status(a.status, BRISK_ERR_INVALID_ARG); rb = 0; }
    const int xb = a.cand_ids[row * K + rb];
    const int xh = a.head_tokens[row];
    int rh = -1;
    for (int k = 0; k < K; ++k)
      if (a.cand_ids[row * K + k] == xh) { rh = k; break; }
    if (rh < 0 || xb < 0 || xb >= a.V || xh < 0 || xh >= a.V) { set_status(a.status, BRISK_ERR_INVALID_ARG); continue; }
    const float lse = a.lse_p[row];
    const float u = a.u_acc[row];
    // alpha = min(1, p(x) / q(x)) = min(1, exp(log p(x) - log q(x)))
    const float ab = fminf(1.f, expf(logit_at(a.logits_p, a.logits_dt, row * a.V + xb) - lse -
                                     a.cand_logprob[row * K + rb]));
    const float ah = fminf(1.f, expf(logit_at(a.logits_p, a.logits_dt, row * a.V + xh) - lse -
                                     a.cand_logprob[row * K + rh]));
    jb[h] = u < ab;
    jh[h] = u < ah;
    changed[h] = xh != xb;
  }
  // first breaker: lowest position whose base token is rejected
  const unsigned rej0 = __ballot_sync(FULL_MASK, lane < L && !jb[0]);
  const unsigned rej1 = __ballot_sync(FULL_MASK, lane + 32 < L && !jb[1]);
  const int fb = rej0 ? __ffs(rej0) - 1 : (rej1 ? 32 + __ffs(rej1) - 1 : L);
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    if (i >= L) continue;
    int f = (jb[h] ? 1 : 0) | (jh[h] ? 2 : 0) | (i == fb ? 4 : 0) | (changed[h] ? 8 : 0);
    if (i == fb && jh[h]) f |= 16;    // rescue
    if (i < fb && !jh[h]) f |= 32;    // regression
    a.flags[(size_t)b * L + i] = f;
  }
  if (lane == 0) a.first_breaker[b] = fb;
}

}  // namespace

cudaError_t launch_replay(const ReplayArgs& a, cudaStream_t stream) {
  const int grid = (a.B + REPLAY_WARPS - 1) / REPLAY_WARPS;
  replay_kernel<<<grid, REPLAY_WARPS * 32, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace brisk
