// Vocabulary sweep: per logit row, the log-partition and the ordered top-K
// (Sec. 3.3 "C_i = TopK(q_i, K)"; App. C.3 ordered candidate set), and for
// verifier rows the argmax (lowest id on ties) and the log-partition.
//
// Work unit: one warp sweeps one chunk of one row with coalesced 16-byte
// streaming loads, SWEEP_UNROLL in flight per lane. Each lane keeps a running
// (max, sum of exp) pair. The warp keeps one exact best-first list of the
// chunk's top-K (logit, id) pairs spread over its lanes (lane k holds the
// k-th best) and a warp-uniform threshold T, a lower bound on the K-th best
// so far: a 16-byte vector whose max is below T cannot contribute, so the
// common case costs one compare per vector. The rare vectors that reach T are
// broadcast to the whole warp and their elements inserted cooperatively.
// The warps of a CTA either sweep different rows or split one row (the two
// layouts of sweep_kernel). Partial results of one row are merged in chunk
// order, in shared memory within a CTA and otherwise through the workspace
// by the last warp to finish the row (arrival counter, no waiting), so
// results do not depend on timing.
#include "brisk_internal.cuh"

namespace brisk {

namespace {

constexpr int SWEEP_WARPS = 4;                 // warps of a split-layout CTA (and the most)
constexpr int SWEEP_ROW_WARPS = 2;             // warps of a row-layout CTA: small CTAs pack
                                               // around a concurrent kernel's CTAs
constexpr int SWEEP_UNROLL = 8;                // 16-byte loads in flight per lane
constexpr int SWEEP_TARGET_TASKS = 152 * 16;   // warp tasks per tensor the chunking aims for
constexpr int SWEEP_MIN_VEC_PER_LANE = 32;
constexpr int SWEEP_CHUNK_VEC = 4096;          // 16-byte vectors a split-layout chunk (64 KB)

// Online log-sum-exp of one group of N logits whose max is mx.
template <int N>
__device__ __forceinline__ void lse_update(const float (&f)[N], float mx, float& m, float& s) {
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
}

template <int N>
__device__ __forceinline__ float max_of(const float (&f)[N]) {
  float mx = f[0];
#pragma unroll
  for (int j = 1; j < N; ++j) mx = fmaxf(mx, f[j]);
  return mx;
}

// Warp list: lane k < kout holds the k-th best (wv, wi); the other lanes hold (-inf, INVALID).
// Cooperative insertion of (v, id), identical in every lane; returns the new K-th value.
__device__ __forceinline__ float wlist_insert(float v, int id, float& wv, int& wi, int kout) {
  const int lane = threadIdx.x & 31;
  const bool ahead = lane < kout && !better(v, id, wv, wi);     // entries that stay before it
  const int pos = __popc(__ballot_sync(FULL_MASK, ahead));
  const float uv = __shfl_up_sync(FULL_MASK, wv, 1);
  const int ui = __shfl_up_sync(FULL_MASK, wi, 1);
  if (pos < kout && lane < kout) {
    if (lane == pos) { wv = v; wi = id; }
    else if (lane > pos) { wv = uv; wi = ui; }
  }
  return __shfl_sync(FULL_MASK, wv, kout - 1);
}

// k-th largest (k in 1..32) of one float per lane, the same in every lane (bitonic sort).
__device__ __forceinline__ float warp_kth_largest(float x, int k) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int j = size >> 1; j > 0; j >>= 1) {
      const float y = __shfl_xor_sync(FULL_MASK, x, j);
      const bool ascending = (lane & size) == 0;
      const bool lower = (lane & j) == 0;
      x = (lower == ascending) ? fminf(x, y) : fmaxf(x, y);
    }
  }
  return __shfl_sync(FULL_MASK, x, 32 - k);
}

// The rare path, for one vector slot u in which some lane's vector reaches T. Every lane has
// written its vector u to the warp's buffer in shared memory; vector u of lane l holds ids
// id0(l) + u * 32 * VN + j. Each vector whose max (mx, per lane) reaches T is read by the whole
// warp (a broadcast from shared memory) and its elements at or above T are inserted in id
// order. offer_vector_call keeps one out-of-line copy of the insertion code; inlined into the
// unrolled loop it costs no register saves around a call (which spilled at the 64-register
// cap), which the row layout's many top-K offers per row repay (measured alone on the
// 128 x 32 x 126464 proposal rows: 188 -> 175 us).
template <typename T>
__device__ __forceinline__ void offer_vector(const uint4* warp_buf, float mx, int id0_lane, int u,
                                             float& thr, float& wv, int& wi, int kout) {
  constexpr int VN = Vec<T>::N;
  const int lane = threadIdx.x & 31;
  unsigned trig = __ballot_sync(FULL_MASK, mx >= thr);
  while (trig) {
    const int src = __ffs(trig) - 1;
    trig &= trig - 1;
    // lane j < VN reads element j of lane src's vector
    const T* e = reinterpret_cast<const T*>(warp_buf + src);
    const float g = lane < VN ? to_f32(e[lane]) : -INFINITY;
    const int id0 = __shfl_sync(FULL_MASK, id0_lane, src) + u * 32 * VN;
    unsigned em = __ballot_sync(FULL_MASK, lane < VN && g >= thr);
    while (em) {
      const int j = __ffs(em) - 1;
      em &= em - 1;
      const float gj = __shfl_sync(FULL_MASK, g, j);
      if (gj >= thr) thr = fmaxf(thr, wlist_insert(gj, id0 + j, wv, wi, kout));
    }
  }
}

template <typename T>
__device__ __noinline__ void offer_vector_call(const uint4* warp_buf, float mx, int id0_lane, int u,
                                               float& thr, float& wv, int& wi, int kout) {
  offer_vector<T>(warp_buf, mx, id0_lane, u, thr, wv, wi, kout);
}

// One scalar element per lane (head or tail of a row), offered like a vector.
__device__ __forceinline__ void offer_scalars(float f, int id, float& thr, float& wv, int& wi,
                                              int kout) {
  unsigned trig = __ballot_sync(FULL_MASK, f >= thr);
  while (trig) {
    const int src = __ffs(trig) - 1;
    trig &= trig - 1;
    const float g = __shfl_sync(FULL_MASK, f, src);
    const int gid = __shfl_sync(FULL_MASK, id, src);
    if (g >= thr) thr = fmaxf(thr, wlist_insert(g, gid, wv, wi, kout));
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

// Max of the VN logits of one 16-byte vector (bf16 pairs compared packed: 3 instructions).
__device__ __forceinline__ float vec_max(const uint4& w, __nv_bfloat16) {
  const __nv_bfloat162 a = __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&w.x),
                                   *reinterpret_cast<const __nv_bfloat162*>(&w.y));
  const __nv_bfloat162 b = __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&w.z),
                                   *reinterpret_cast<const __nv_bfloat162*>(&w.w));
  const __nv_bfloat162 c = __hmax2(a, b);
  return fmaxf(__low2float(c), __high2float(c));
}
__device__ __forceinline__ float vec_max(const uint4& w, float) {
  return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
               fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
}

// Per-lane state of a chunk sweep.
struct ChunkState {
  float m, s;      // running max and sum of exp(x - max)
  float wv;        // warp list entry held by this lane
  int wi;
  float thr;       // warp-uniform lower bound on the K-th best so far
  bool first;
};

// One iteration: SWEEP_UNROLL vectors per lane, lane's vector u holding ids
// head + (base + lane + 32 u) * VN + j. The running max moves once per iteration, so all of the
// iteration's exponentials share one offset; arguments and sums use packed fp32 pairs.
// INLINE_OFFER: the rare offer path inlined (row layout) or called (split layout).
template <typename T, bool INLINE_OFFER>
__device__ __forceinline__ void sweep_iteration(const uint4 (&w)[SWEEP_UNROLL], int id0_lane,
                                                int kout, uint4* warp_buf, ChunkState& st) {
  constexpr int VN = Vec<T>::N;
  float mx[SWEEP_UNROLL];
  float mx_all = -INFINITY;
#pragma unroll
  for (int u = 0; u < SWEEP_UNROLL; ++u) {
    mx[u] = vec_max(w[u], T());
    mx_all = fmaxf(mx_all, mx[u]);
  }
  if (mx_all > st.m) {
    st.s *= ex2((st.m - mx_all) * LOG2E);
    st.m = mx_all;
  }
  if (st.m != -INFINITY) {
    const float nmb = -st.m * LOG2E;
    const float2 l2e = make_float2(LOG2E, LOG2E), off = make_float2(nmb, nmb);
    float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
    for (int u = 0; u < SWEEP_UNROLL; ++u) {
      float f[VN];
      unpack(w[u], f, T());
#pragma unroll
      for (int j = 0; j < VN; j += 2) {
        const float2 arg = __ffma2_rn(make_float2(f[j], f[j + 1]), l2e, off);
        const float2 e = make_float2(ex2(arg.x), ex2(arg.y));
        if ((j / 2 + u) & 1) acc1 = __fadd2_rn(acc1, e);
        else acc0 = __fadd2_rn(acc0, e);
      }
    }
    const float2 acc = __fadd2_rn(acc0, acc1);
    st.s += acc.x + acc.y;
  }
  if (st.first) {
    // K lanes each hold an element at least this large: a lower bound on the K-th best
    st.thr = fmaxf(st.thr, warp_kth_largest(mx_all, kout));
    st.first = false;
  }
  unsigned umask = 0;
#pragma unroll
  for (int u = 0; u < SWEEP_UNROLL; ++u) umask |= (mx[u] >= st.thr ? 1u : 0u) << u;
  umask = __reduce_or_sync(FULL_MASK, umask);
  if (umask) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int u = 0; u < SWEEP_UNROLL; ++u) {
      if (umask & (1u << u)) {
        warp_buf[lane] = w[u];
        __syncwarp();
        if constexpr (INLINE_OFFER)
          offer_vector<T>(warp_buf, mx[u], id0_lane, u, st.thr, st.wv, st.wi, kout);
        else
          offer_vector_call<T>(warp_buf, mx[u], id0_lane, u, st.thr, st.wv, st.wi, kout);
        __syncwarp();
      }
    }
  }
}

// One warp's sweep of chunk `chunk` (of nchunk) of the row at rowp: on return every lane holds
// the chunk's (max, sum of exp) pair and the warp list holds its best-first top-kout.
template <typename T, bool INLINE_OFFER>
__device__ __forceinline__ void sweep_chunk(const T* rowp, int V, int chunk, int nchunk, int kout,
                                            uint4* warp_buf, float& m, float& s, float& wv,
                                            int& wi) {
  constexpr int VN = Vec<T>::N;
  constexpr int STEP = 32 * SWEEP_UNROLL;
  const int lane = threadIdx.x & 31;
  const uintptr_t addr = reinterpret_cast<uintptr_t>(rowp);
  int head = (int)(((16u - (unsigned)(addr & 15u)) & 15u) / sizeof(T));
  if (head > V) head = V;
  const int nvec = (V - head) / VN;
  const int tail0 = head + nvec * VN;
  const int vpc = (nvec + nchunk - 1) / nchunk;
  const int v_begin = chunk * vpc;
  const int v_end = min(nvec, v_begin + vpc);

  ChunkState st{-INFINITY, 0.f, -INFINITY, INVALID_ID, -INFINITY, true};

  // unaligned head (ids below every vector): lanes 0..head-1 of chunk 0
  if (chunk == 0) {
    float f = -INFINITY;
    if (lane < head) {
      f = to_f32(rowp[lane]);
      const float ff[1] = {f};
      lse_update<1>(ff, f, st.m, st.s);
    }
    offer_scalars(f, lane < head ? lane : INVALID_ID, st.thr, st.wv, st.wi, kout);
  }
  const uint4* vp = reinterpret_cast<const uint4*>(rowp + head);
  int base = v_begin;
  // full iterations: no bounds checks
  for (; base + STEP <= v_end; base += STEP) {
    uint4 w[SWEEP_UNROLL];
#pragma unroll
    for (int u = 0; u < SWEEP_UNROLL; ++u) w[u] = ld_stream_v4(vp + base + lane + 32 * u);
    sweep_iteration<T, INLINE_OFFER>(w, head + (base + lane) * VN, kout, warp_buf, st);
  }
  // the ragged last iteration, padded with -inf
  if (base < v_end) {
    const uint32_t ninf = VN == 8 ? 0xff80ff80u : 0xff800000u;
    uint4 w[SWEEP_UNROLL];
#pragma unroll
    for (int u = 0; u < SWEEP_UNROLL; ++u) {
      const int v = base + lane + 32 * u;
      w[u] = v < v_end ? ld_stream_v4(vp + v) : make_uint4(ninf, ninf, ninf, ninf);
    }
    sweep_iteration<T, INLINE_OFFER>(w, head + (base + lane) * VN, kout, warp_buf, st);
  }
  // ragged tail (ids above every vector): lanes of the last chunk, one element each
  if (chunk == nchunk - 1) {
    const int e = tail0 + lane;
    float f = -INFINITY;
    if (e < V) {
      f = to_f32(rowp[e]);
      const float ff[1] = {f};
      lse_update<1>(ff, f, st.m, st.s);
    }
    offer_scalars(f, e < V ? e : INVALID_ID, st.thr, st.wv, st.wi, kout);
  }
  warp_lse_combine(st.m, st.s);
  m = st.m;
  s = st.s;
  wv = st.wv;
  wi = st.wi;
}

// Publishes one partial result (part index pb of the row) and, in the last of the row's
// `parts` warps to arrive (arrival counter, no waiting), merges all of them in part order and
// writes the row's outputs. Called by one whole warp.
__device__ __forceinline__ void publish_partial(const SweepSeg& sg, int row, int pb_in_row,
                                                int parts, int KP, float m, float s, float wv,
                                                int wi, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int kout = sg.kout;
  const size_t pb = (size_t)row * parts + pb_in_row;
  if (lane < kout) {
    sg.part_val[pb * KP + lane] = wv;
    sg.part_id[pb * KP + lane] = wi;
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
  if (prev != parts - 1) return;
  __threadfence();

  // last part of the row: merge the partials in part order, the lists of MERGE_BATCH parts
  // loaded at once (one L2 round trip per batch instead of one per part)
  constexpr int MERGE_BATCH = 8;
  wv = -INFINITY;
  wi = INVALID_ID;
  float thr = -INFINITY;
  for (int c0 = 0; c0 < parts; c0 += MERGE_BATCH) {
    float f[MERGE_BATCH];
    int id[MERGE_BATCH];
#pragma unroll
    for (int u = 0; u < MERGE_BATCH; ++u) {
      f[u] = -INFINITY;
      id[u] = INVALID_ID;
      if (c0 + u < parts && lane < kout) {
        const size_t q = ((size_t)row * parts + c0 + u) * KP;
        f[u] = __ldcg(sg.part_val + q + lane);
        id[u] = __ldcg(sg.part_id + q + lane);
      }
    }
#pragma unroll
    for (int u = 0; u < MERGE_BATCH; ++u) offer_scalars(f[u], id[u], thr, wv, wi, kout);
  }
  float mm = -INFINITY, ss = 0.f;
  for (int c = lane; c < parts; c += 32) {
    const size_t q = (size_t)row * parts + c;
    lse_merge(mm, ss, __ldcg(sg.part_m + q), __ldcg(sg.part_s + q));
  }
  warp_lse_combine(mm, ss);
  finalize_row(sg, row, mm, ss, wv, wi, status);
  if (lane == 0) sg.counters[row] = 0;
}

// Two work layouts (SweepLaunch::mode):
//  SWEEP_ROWS : each warp sweeps its own (row, chunk) task; a CTA holds blockDim / 32 tasks.
//               One warp sees a whole row when the row is not split, so the top-K threshold
//               tightens over the whole row (the proposal rows' layout).
//  SWEEP_SPLIT: a CTA sweeps one (row, split): its warps take consecutive chunks and merge in
//               shared memory. Many short CTAs let the block scheduler balance the work over
//               SMs that a concurrent kernel slows down (the verifier rows' layout, which runs
//               beside the corrector).
// At most 64 registers a thread: eight 4-warp CTAs fit an SM's register file, so a full wave
// of the sweep still fits beside a CTA of a concurrent kernel.
template <typename T, int MODE>
__global__ void __launch_bounds__(SWEEP_WARPS * 32, 8)
sweep_kernel(const __grid_constant__ SweepLaunch a) {
  __shared__ uint4 stash[SWEEP_WARPS * 32];
  __shared__ float mvals[SWEEP_WARPS][32];
  __shared__ int mids[SWEEP_WARPS][32];
  __shared__ float mms[SWEEP_WARPS][2];
  const int nw = blockDim.x >> 5;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint4* warp_buf = stash + warp * 32;
  const int V = a.V;

  if constexpr (MODE == SWEEP_ROWS) {
    const long long task = (long long)blockIdx.x * nw + warp;
    const long long tasks0 = (long long)a.seg[0].rows * a.nchunk;
    const long long total = tasks0 + (a.nseg > 1 ? (long long)a.seg[1].rows * a.nchunk : 0);
    if (task >= total) return;
    const int si = task < tasks0 ? 0 : 1;
    const SweepSeg& sg = a.seg[si];
    const long long t = si ? task - tasks0 : task;
    const int row = (int)(t / a.nchunk);
    const int chunk = (int)(t % a.nchunk);
    const T* rowp = reinterpret_cast<const T*>(sg.logits) + (size_t)row * V;
    float m, s, wv;
    int wi;
    sweep_chunk<T, true>(rowp, V, chunk, a.nchunk, sg.kout, warp_buf, m, s, wv, wi);
    if (a.nchunk == 1) finalize_row(sg, row, m, s, wv, wi, a.status);
    else publish_partial(sg, row, chunk, a.nchunk, a.KP, m, s, wv, wi, a.status);
    return;
  } else {

  const int nsplit = a.nchunk / nw;                     // CTAs per row
  const long long ctas0 = (long long)a.seg[0].rows * nsplit;
  const long long cta = blockIdx.x;
  const int si = cta < ctas0 ? 0 : 1;
  const SweepSeg& sg = a.seg[si];
  const long long t = si ? cta - ctas0 : cta;
  const int row = (int)(t / nsplit);
  const int split = (int)(t % nsplit);
  const int kout = sg.kout;
  const T* rowp = reinterpret_cast<const T*>(sg.logits) + (size_t)row * V;
  float m, s, wv;
  int wi;
  sweep_chunk<T, false>(rowp, V, split * nw + warp, a.nchunk, kout, warp_buf, m, s, wv, wi);
  // the CTA's warps merged by warp 0 in chunk order
  mvals[warp][lane] = wv;
  mids[warp][lane] = wi;
  if (lane == 0) {
    mms[warp][0] = m;
    mms[warp][1] = s;
  }
  __syncthreads();
  if (warp != 0) return;
  float thr = -INFINITY;
  for (int w = 1; w < nw; ++w) {
    offer_scalars(lane < kout ? mvals[w][lane] : -INFINITY, lane < kout ? mids[w][lane] : INVALID_ID,
                  thr, wv, wi, kout);
    lse_merge(m, s, mms[w][0], mms[w][1]);
  }
  if (nsplit == 1) finalize_row(sg, row, m, s, wv, wi, a.status);
  else publish_partial(sg, row, split, nsplit, a.KP, m, s, wv, wi, a.status);
  }
}

template <typename T>
cudaError_t launch_t(const SweepLaunch& a, cudaStream_t stream) {
  long long rows = a.seg[0].rows;
  if (a.nseg > 1) rows += a.seg[1].rows;
  if (a.mode == SWEEP_ROWS) {
    const long long tasks = rows * a.nchunk;
    const unsigned grid = (unsigned)((tasks + SWEEP_ROW_WARPS - 1) / SWEEP_ROW_WARPS);
    cudaError_t e = prefer_carveout(sweep_kernel<T, SWEEP_ROWS>, CARVEOUT_SMALL_KB);
    if (e != cudaSuccess) return e;
    e = launch_prio(sweep_kernel<T, SWEEP_ROWS>, dim3(grid), dim3(SWEEP_ROW_WARPS * 32), 0, stream, a);
    if (e != cudaSuccess) return e;
  } else {
    const unsigned grid = (unsigned)(rows * (a.nchunk / SWEEP_WARPS));
    cudaError_t e = prefer_carveout(sweep_kernel<T, SWEEP_SPLIT>, CARVEOUT_SMALL_KB);
    if (e != cudaSuccess) return e;
    e = launch_prio(sweep_kernel<T, SWEEP_SPLIT>, dim3(grid), dim3(SWEEP_WARPS * 32), 0, stream, a);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

}  // namespace

int kp_for(int K) {
  int kp = 4;
  while (kp < K) kp *= 2;
  return kp;
}

// Chunks per row. Independent of the device so that the summation order, and hence every
// rounded result, is the same on every run.
//  SWEEP_ROWS : enough warp tasks per tensor to keep every SM streaming, but at least
//               SWEEP_MIN_VEC_PER_LANE 16-byte vectors per lane.
//  SWEEP_SPLIT: a multiple of SWEEP_WARPS, about SWEEP_CHUNK_VEC vectors a chunk, and enough
//               CTAs per tensor to keep every SM streaming.
int sweep_chunks(int rows_per_tensor, int V, int dtype, int mode) {
  const int vn = dtype == BRISK_DT_BF16 ? 8 : 4;
  const long long nvec = V / vn;
  if (mode == SWEEP_ROWS) {
    long long maxc = nvec / (32LL * SWEEP_MIN_VEC_PER_LANE);
    if (maxc < 1) maxc = 1;
    long long c = (SWEEP_TARGET_TASKS + rows_per_tensor - 1) / rows_per_tensor;
    if (c < 1) c = 1;
    if (c > maxc) c = maxc;
    return (int)c;
  }
  long long maxs = nvec / (32LL * SWEEP_MIN_VEC_PER_LANE * SWEEP_WARPS);
  if (maxs < 1) maxs = 1;
  const long long target = (SWEEP_TARGET_TASKS + SWEEP_WARPS - 1) / SWEEP_WARPS;
  long long c = (target + rows_per_tensor - 1) / rows_per_tensor;
  const long long per_cta = (long long)SWEEP_CHUNK_VEC * SWEEP_WARPS;
  const long long by_size = (nvec + per_cta - 1) / per_cta;
  if (c < by_size) c = by_size;
  if (c < 1) c = 1;
  if (c > maxs) c = maxs;
  return (int)c * SWEEP_WARPS;
}

cudaError_t launch_sweep(const SweepLaunch& a, cudaStream_t stream) {
  if (a.dtype == BRISK_DT_BF16) return launch_t<__nv_bfloat16>(a, stream);
  return launch_t<float>(a, stream);
}

}  // namespace brisk
