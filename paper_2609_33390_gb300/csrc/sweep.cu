// Vocabulary sweep: per logit row, the log-partition and the ordered top-K
// (Sec. 3.3 "C_i = TopK(q_i, K)"; App. C.2 ordered candidate set), and for
// verifier rows the argmax (lowest id on ties) and the log-partition.
//
// Work unit: one warp sweeps one chunk of one row with coalesced 16-byte
// streaming loads. Each lane keeps a running (max, sum of exp) pair and a
// best-first list of KP >= K (logit, id) entries in registers; an element
// costs one max, one exp and one add, and enters the list only when it beats
// the list's last entry. The warp then merges its 32 lists and pairs. When a
// row is split into several chunks, each warp writes its partial result to
// the workspace and the last warp to finish the row (arrival counter)
// merges the partials in chunk order, so results do not depend on timing.
#include "brisk_internal.cuh"

namespace brisk {

namespace {

constexpr int SWEEP_WARPS = 4;            // independent warps per CTA
constexpr int SWEEP_TARGET_TASKS = 152 * 48;  // warp tasks per tensor the chunking aims for
constexpr int SWEEP_MIN_VEC_PER_LANE = 8;

template <int KP, int N>
__device__ __forceinline__ void consume(const float (&f)[N], int id0, float& m, float& s,
                                        float (&vals)[KP], int (&ids)[KP]) {
  float mx = f[0];
#pragma unroll
  for (int j = 1; j < N; ++j) mx = fmaxf(mx, f[j]);
  if (mx > m) {
    s *= ex2((m - mx) * LOG2E);
    m = mx;
  }
  if (m != -INFINITY) {
    const float mb = m * LOG2E;
    float a0 = 0.f, a1 = 0.f;
#pragma unroll
    for (int j = 0; j < N; j += 2) {
      a0 += ex2(fmaf(f[j], LOG2E, -mb));
      if (j + 1 < N) a1 += ex2(fmaf(f[j + 1], LOG2E, -mb));
    }
    s += a0 + a1;
  }
  if (mx >= vals[KP - 1]) {
#pragma unroll
    for (int j = 0; j < N; ++j)
      if (better(f[j], id0 + j, vals[KP - 1], ids[KP - 1])) list_insert<KP>(f[j], id0 + j, vals, ids);
  }
}

__device__ __forceinline__ void lse_merge(float& m, float& s, float pm, float ps) {
  if (pm == -INFINITY) return;
  if (m == -INFINITY) {
    m = pm;
    s = ps;
  } else if (pm > m) {
    s = s * ex2((m - pm) * LOG2E) + ps;
    m = pm;
  } else {
    s += ps * ex2((pm - m) * LOG2E);
  }
}

__device__ __forceinline__ void finalize_row(const SweepSeg& sg, int row, float M, float S,
                                             float ov, int oi, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const float lse = M + logf(S);
  if (!isfinite(lse) && lane == 0) set_status(status, BRISK_ERR_NUMERIC);
  if (lane < sg.kout) {
    sg.out_ids[(size_t)row * sg.kout + lane] = oi;
    if (sg.out_logprob) sg.out_logprob[(size_t)row * sg.kout + lane] = ov - lse;
  }
  if (lane == 0) sg.out_lse[row] = lse;
}

template <typename T, int KP>
__global__ void __launch_bounds__(SWEEP_WARPS * 32)
sweep_kernel(const __grid_constant__ SweepLaunch a) {
  constexpr int VN = Vec<T>::N;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const long long task = (long long)blockIdx.x * SWEEP_WARPS + warp;
  const long long tasks0 = (long long)a.seg[0].rows * a.nchunk;
  const long long total = tasks0 + (a.nseg > 1 ? (long long)a.seg[1].rows * a.nchunk : 0);
  if (task >= total) return;
  const int si = task < tasks0 ? 0 : 1;
  const SweepSeg& sg = a.seg[si];
  const long long t = si ? task - tasks0 : task;
  const int row = (int)(t / a.nchunk);
  const int chunk = (int)(t % a.nchunk);
  const int V = a.V;

  const T* rowp = reinterpret_cast<const T*>(sg.logits) + (size_t)row * V;
  const uintptr_t addr = reinterpret_cast<uintptr_t>(rowp);
  int head = (int)(((16u - (unsigned)(addr & 15u)) & 15u) / sizeof(T));
  if (head > V) head = V;
  const int nvec = (V - head) / VN;
  const int tail0 = head + nvec * VN;
  const int vpc = (nvec + a.nchunk - 1) / a.nchunk;
  const int v_begin = chunk * vpc;
  const int v_end = min(nvec, v_begin + vpc);

  float m = -INFINITY, s = 0.f;
  float vals[KP];
  int ids[KP];
  list_clear<KP>(vals, ids);

  // unaligned head (ids below every vector): lane 0 of chunk 0
  if (chunk == 0 && lane == 0) {
    for (int e = 0; e < head; ++e) {
      const float f[1] = {to_f32(rowp[e])};
      consume<KP, 1>(f, e, m, s, vals, ids);
    }
  }
  const uint4* vp = reinterpret_cast<const uint4*>(rowp + head);
  int v = v_begin + lane;
  for (; v + 96 < v_end; v += 128) {
    const uint4 w0 = ld_stream_v4(vp + v);
    const uint4 w1 = ld_stream_v4(vp + v + 32);
    const uint4 w2 = ld_stream_v4(vp + v + 64);
    const uint4 w3 = ld_stream_v4(vp + v + 96);
    float f[VN];
    unpack(w0, f, T());
    consume<KP, VN>(f, head + v * VN, m, s, vals, ids);
    unpack(w1, f, T());
    consume<KP, VN>(f, head + (v + 32) * VN, m, s, vals, ids);
    unpack(w2, f, T());
    consume<KP, VN>(f, head + (v + 64) * VN, m, s, vals, ids);
    unpack(w3, f, T());
    consume<KP, VN>(f, head + (v + 96) * VN, m, s, vals, ids);
  }
  for (; v < v_end; v += 32) {
    const uint4 w0 = ld_stream_v4(vp + v);
    float f[VN];
    unpack(w0, f, T());
    consume<KP, VN>(f, head + v * VN, m, s, vals, ids);
  }
  // ragged tail (ids above every vector): last chunk, one element per lane
  if (chunk == a.nchunk - 1) {
    const int e = tail0 + lane;
    if (e < V) {
      const float f[1] = {to_f32(rowp[e])};
      consume<KP, 1>(f, e, m, s, vals, ids);
    }
  }

  warp_lse_combine(m, s);
  float ov;
  int oi;
  warp_extract<KP>(vals, ids, sg.kout, ov, oi);
  if (a.nchunk == 1) {
    finalize_row(sg, row, m, s, ov, oi, a.status);
    return;
  }

  const size_t pb = (size_t)row * a.nchunk + chunk;
  if (lane < sg.kout) {
    sg.part_val[pb * KP + lane] = ov;
    sg.part_id[pb * KP + lane] = oi;
  }
  if (lane == 0) {
    sg.part_m[pb] = m;
    sg.part_s[pb] = s;
  }
  __threadfence();
  __syncwarp();
  int prev = 0;
  if (lane == 0) prev = atomicAdd(&sg.counters[row], 1);
  prev = __shfl_sync(FULL_MASK, prev, 0);
  if (prev != a.nchunk - 1) return;
  __threadfence();

  // last warp of the row: merge the chunk partials in chunk order
  list_clear<KP>(vals, ids);
  const int nent = a.nchunk * sg.kout;
  for (int e = lane; e < nent; e += 32) {
    const int c = e / sg.kout, k = e - c * sg.kout;
    const size_t q = ((size_t)row * a.nchunk + c) * KP + k;
    list_insert<KP>(__ldcg(sg.part_val + q), __ldcg(sg.part_id + q), vals, ids);
  }
  float mm = -INFINITY, ss = 0.f;
  for (int c = lane; c < a.nchunk; c += 32) {
    const size_t q = (size_t)row * a.nchunk + c;
    lse_merge(mm, ss, __ldcg(sg.part_m + q), __ldcg(sg.part_s + q));
  }
  warp_lse_combine(mm, ss);
  warp_extract<KP>(vals, ids, sg.kout, ov, oi);
  finalize_row(sg, row, mm, ss, ov, oi, a.status);
  if (lane == 0) sg.counters[row] = 0;
}

template <typename T>
cudaError_t launch_t(const SweepLaunch& a, cudaStream_t stream) {
  long long tasks = (long long)a.seg[0].rows * a.nchunk;
  if (a.nseg > 1) tasks += (long long)a.seg[1].rows * a.nchunk;
  const unsigned grid = (unsigned)((tasks + SWEEP_WARPS - 1) / SWEEP_WARPS);
  const dim3 block(SWEEP_WARPS * 32);
  switch (a.KP) {
    case 4: sweep_kernel<T, 4><<<grid, block, 0, stream>>>(a); break;
    case 8: sweep_kernel<T, 8><<<grid, block, 0, stream>>>(a); break;
    case 16: sweep_kernel<T, 16><<<grid, block, 0, stream>>>(a); break;
    case 32: sweep_kernel<T, 32><<<grid, block, 0, stream>>>(a); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

int kp_for(int K) {
  int kp = 4;
  while (kp < K) kp *= 2;
  return kp;
}

// Chunks per row: enough warp tasks per tensor to keep every SM streaming, but at least
// SWEEP_MIN_VEC_PER_LANE 16-byte vectors per lane. Independent of the device so that the
// summation order, and hence every rounded result, is the same on every run.
int sweep_chunks(int rows_per_tensor, int V, int dtype, int /*num_sms*/) {
  const int vn = dtype == BRISK_DT_BF16 ? 8 : 4;
  const long long nvec = V / vn;
  long long maxc = nvec / (32LL * SWEEP_MIN_VEC_PER_LANE);
  if (maxc < 1) maxc = 1;
  long long c = (SWEEP_TARGET_TASKS + rows_per_tensor - 1) / rows_per_tensor;
  if (c < 1) c = 1;
  if (c > maxc) c = maxc;
  return (int)c;
}

cudaError_t launch_sweep(const SweepLaunch& a, cudaStream_t stream) {
  if (a.dtype == BRISK_DT_BF16) return launch_t<__nv_bfloat16>(a, stream);
  return launch_t<float>(a, stream);
}

}  // namespace brisk
