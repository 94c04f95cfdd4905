// Distillation loss of the refinement head and its gradient in the refined scores (App. C.3,
// Eq. 10): at every reached position j of a block (the accepted prefix and the first rejected
// position), CE(p_S, r) + beta KL(q_S || r), with p_S the verifier distribution restricted to
// the candidate set S_j and renormalised, q_S the base distribution restricted to S_j, and
// r = softmax(refined scores); one mean over all reached positions of the batch.
//
// One CTA per sequence, one warp per position (lane k = candidate k). Each CTA writes its
// positions' gradients and its loss sum; the last CTA to finish (arrival counter, no waiting)
// adds the per-sequence sums in sequence order, so the loss does not depend on timing.
#include "brisk_internal.cuh"

namespace brisk {
namespace {

constexpr int DISTILL_WARPS = 4;

__device__ __forceinline__ float load_logit_d(const void* base, int dt, size_t idx) {
  if (dt == BRISK_DT_BF16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(base)[idx]);
  return reinterpret_cast<const float*>(base)[idx];
}

// Softmax over the lanes below K of one value per lane: the probability and its log.
__device__ __forceinline__ void lane_softmax(float x, int K, float& prob, float& logp) {
  const int lane = threadIdx.x & 31;
  const float v = lane < K ? x : -INFINITY;
  const float m = warp_max(v);
  const float e = lane < K ? __expf(v - m) : 0.f;
  const float z = warp_sum(e);
  prob = e / z;
  logp = lane < K ? (v - m) - __logf(z) : -INFINITY;
}

__global__ void __launch_bounds__(DISTILL_WARPS * 32)
distill_kernel(const __grid_constant__ DistillArgs a) {
  __shared__ float pos_loss[64];
  __shared__ int last;
  const int b = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int L = a.L, K = a.K;
  // reached positions of every sequence of the batch (each CTA counts them: no extra pass)
  int n_local = 0;
  for (int s = threadIdx.x; s < a.B; s += blockDim.x) {
    const int acc = a.accepted_len[s];
    n_local += min(max(acc, 0), L - 1) + 1;
  }
  __shared__ int n_warp[DISTILL_WARPS];
  n_local = __reduce_add_sync(FULL_MASK, n_local);
  if (lane == 0) n_warp[warp] = n_local;
  __syncthreads();
  int n_total = 0;
  for (int w = 0; w < DISTILL_WARPS; ++w) n_total += n_warp[w];
  const float inv_n = 1.f / (float)n_total;
  const int reach = min(max(a.accepted_len[b], 0), L - 1);   // positions 0..reach are reached

  for (int j = warp; j < L; j += DISTILL_WARPS) {
    const size_t row = (size_t)b * L + j;
    const size_t e = row * K + lane;
    if (j > reach) {
      if (a.grad && lane < K) a.grad[e] = 0.f;
      if (lane == 0) pos_loss[j] = 0.f;
      continue;
    }
    float pl = -INFINITY, ql = -INFINITY, rl = -INFINITY;
    if (lane < K) {
      int c = a.cand_ids[e];
      if (c < 0 || c >= a.V) { set_status(a.status, BRISK_ERR_INVALID_ARG); c = 0; }
      pl = load_logit_d(a.logits_p, a.logits_dt, row * a.V + c);
      ql = a.cand_logprob[e];
      rl = a.refined[e];
    }
    float p, logp, q, logq, r, logr;
    lane_softmax(pl, K, p, logp);
    lane_softmax(ql, K, q, logq);
    lane_softmax(rl, K, r, logr);
    // terms with zero mass contribute nothing (0 log 0 = 0)
    float term = 0.f;
    if (lane < K) {
      if (p > 0.f) term -= p * logr;
      if (q > 0.f) term += a.beta * q * (logq - logr);
    }
    term = warp_sum(term);
    if (lane == 0) pos_loss[j] = term;
    if (a.grad && lane < K) a.grad[e] = ((r - p) + a.beta * (r - q)) * inv_n;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float sum = 0.f;
    for (int j = 0; j <= reach; ++j) sum += pos_loss[j];
    a.partial[b] = sum;
    __threadfence();
    last = atomicAdd(a.arrivals, 1) == a.B - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    // the last CTA: every partial is visible; add them in sequence order
    float total = 0.f;
    for (int s = 0; s < a.B; ++s) total += __ldcg(a.partial + s);
    a.loss[0] = total * inv_n;
    *a.arrivals = 0;
  }
}

}  // namespace

cudaError_t launch_distill(const DistillArgs& a, cudaStream_t stream) {
  distill_kernel<<<a.B, DISTILL_WARPS * 32, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace brisk
