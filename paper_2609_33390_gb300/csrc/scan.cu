// Corrector scan and verification, one CTA per sequence.
//
// Corrector (Sec. 3.3 Eqs. 4-5; App. C.3 Eq. 9; Algorithm 1(b) loop). The
// minimal-GRU pre-activations are linear in the input blocks
// [P_h m_i ; P_e E_in(x_{i-1}) ; pos_i ; P_phi phi_i], so each block's share is
// read from a precomputed source:
//   hidden share   G[b,i]          (one dense product over all b, i, before the scan)
//   token share    Tzh[x_{i-1}]    (vocabulary table folded once per weight set)
//   position share posz[i], posh[i]
//   feature share  Fz phi_i, Fh phi_i   (S x 5 folded matrices)
// and the residual d_{i,k} = <W_s s_i, W_c E_out(c)> = <s_i, U[c]> with
// U = (E_out W_c^T) W_s. Init is u_0 = tanh(G0[b] + T0[x0]). What stays
// sequential per position is O(S) element work, K+1 dot products of length S
// and the K-way Select.
//
// Verification (Sec. 3.1; Sec. 3.3; App. B Eq. 6) runs in the same CTA after
// the scan, or alone (brisk_verify_block), through the same device code.
#include "brisk_internal.cuh"

namespace brisk {

namespace {

// Verification CTA: 128 threads, or 512 under stochastic verification, where a rejection
// resamples from a residual over the whole vocabulary row (a 126464-entry row: 112 us on 128
// threads with element loads and the precise exponential, a few us with 512 threads, vector
// loads and the hardware one).
constexpr int VERIFY_THREADS = 128;
constexpr int VERIFY_THREADS_MAX = 512;

struct Smem {
  int* cid;        // [L][K]
  int* sel;        // [L]
  int* rank;       // [L]
  float* ref;      // [L][K]
  float* bsum;     // [nblk]  residual block sums
  float* misc;     // [16]
  int* imisc;      // [16]
};

__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

constexpr int RES_BLOCK = 256;  // residual-sampling block: 32 lanes x 8 ids

__host__ __device__ inline size_t smem_layout(int L, int K, int S, int V, char* base, Smem* sm) {
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align16(off + bytes);
    return base ? base + o : nullptr;
  };
  (void)S;
  const int nblk = (V + RES_BLOCK - 1) / RES_BLOCK;
  char* p_cid = take(sizeof(int) * L * K);
  char* p_sel = take(sizeof(int) * L);
  char* p_rank = take(sizeof(int) * L);
  char* p_ref = take(sizeof(float) * L * K);
  char* p_bsum = take(sizeof(float) * nblk);
  char* p_misc = take(sizeof(float) * 16);
  char* p_imisc = take(sizeof(int) * 16);
  if (sm) {
    sm->cid = (int*)p_cid; sm->sel = (int*)p_sel; sm->rank = (int*)p_rank; sm->ref = (float*)p_ref;
    sm->bsum = (float*)p_bsum; sm->misc = (float*)p_misc; sm->imisc = (int*)p_imisc;
  }
  return off;
}

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }

// A lane's chunk of CW consecutive state elements (CW = 1, 2 or 4), loaded as one vector;
// CG: cached in L2 only (rows read once per step must not displace the L1 lines that hold a
// concurrent streaming kernel's loads in flight).
template <int CW>
struct Chunk {
  float v[CW];
};
template <int CW>
__device__ __forceinline__ Chunk<CW> chunk_of(const float4& t) {
  if constexpr (CW == 4) return {{t.x, t.y, t.z, t.w}};
  else return {{t.x, t.y}};
}
template <int CW, bool CG>
__device__ __forceinline__ Chunk<CW> ldc(const float* p) {
  if constexpr (CW == 4) {
    return chunk_of<4>(CG ? __ldcg(reinterpret_cast<const float4*>(p))
                          : *reinterpret_cast<const float4*>(p));
  } else if constexpr (CW == 2) {
    const float2 t = CG ? __ldcg(reinterpret_cast<const float2*>(p))
                        : *reinterpret_cast<const float2*>(p);
    return {{t.x, t.y}};
  } else {
    return {{CG ? __ldcg(p) : *p}};
  }
}
template <int CW>
__device__ __forceinline__ Chunk<CW> addc(const Chunk<CW>& x, const Chunk<CW>& y) {
  Chunk<CW> r;
#pragma unroll
  for (int e = 0; e < CW; ++e) r.v[e] = x.v[e] + y.v[e];
  return r;
}
// acc + sum_e x_e y_e, the last element first (the order of the four-element form)
template <int CW>
__device__ __forceinline__ float dotc(const Chunk<CW>& x, const Chunk<CW>& y, float acc) {
#pragma unroll
  for (int e = CW - 1; e >= 0; --e) acc = fmaf(x.v[e], y.v[e], acc);
  return acc;
}
// Logistic function with the hardware exponential (relative error ~1e-6).
__device__ __forceinline__ float sigmoid_fast(float x) { return __fdividef(1.f, 1.f + __expf(-x)); }

// Warp reduce-scatter of NP values per lane: afterwards lane l holds the warp-wide sum of value
// ((l >> 1) & 15) for NP = 16 and of value l for NP = 32.
template <int NP>
__device__ __forceinline__ float reduce_scatter(float (&v)[NP]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int m = 16, n = NP; n > 1; m >>= 1, n >>= 1) {
    const bool upper = (lane & m) != 0;
#pragma unroll
    for (int j = 0; j < n / 2; ++j) {
      const float send = upper ? v[j] : v[j + n / 2];
      const float keep = upper ? v[j + n / 2] : v[j];
      v[j] = keep + __shfl_xor_sync(FULL_MASK, send, m);
    }
  }
  float r = v[0];
  if (NP == 16) r += __shfl_xor_sync(FULL_MASK, r, 1);
  return r;
}

__device__ __forceinline__ float load_logit(const void* base, int dt, size_t idx) {
  if (dt == BRISK_DT_BF16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(base)[idx]);
  return reinterpret_cast<const float*>(base)[idx];
}

// Order-preserving map of a float (not NaN) to an unsigned key; -0 and +0 map alike.
__device__ __forceinline__ unsigned ordered_key(float f) {
  const unsigned u = __float_as_uint(f + 0.f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_value(unsigned k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Select with lane k holding refined score k (lanes >= K hold -inf); the same in every lane.
// Greedy: argmax, the lowest rank on ties. Sample: the first rank whose cumulative softmax mass
// exceeds u * total (warp prefix sums), else the last rank with mass. The maxima are single
// warp reductions of the scores' order-preserving keys (five shuffle rounds before: single
// 102 -> 100 us, large_vocab 246 -> 241 us for the products and the corrector).
__device__ __forceinline__ int select_warp(float ref, int K, int mode, float u) {
  const int lane = threadIdx.x & 31;
  if (mode == BRISK_SELECT_GREEDY) {
    // a NaN score ranks as -inf, so every lane agrees on one rank in [0, K) whatever the
    // scores hold: the lowest rank holding the warp's largest key (one warp reduction)
    const float bv = (lane < K && !isnan(ref)) ? ref : -INFINITY;
    const unsigned key = ordered_key(bv);
    const unsigned mk = __reduce_max_sync(FULL_MASK, key);
    const unsigned hit = __ballot_sync(FULL_MASK, lane < K && key == mk);
    return hit ? __ffs(hit) - 1 : 0;
  }
  const float mx = key_value(__reduce_max_sync(FULL_MASK, ordered_key(isnan(ref) ? -INFINITY : ref)));
  const float w = lane < K ? expf(ref - mx) : 0.f;
  float cum = w;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float o = __shfl_up_sync(FULL_MASK, cum, off);
    if (lane >= off) cum += o;
  }
  const float tot = __shfl_sync(FULL_MASK, cum, 31);
  const unsigned hit = __ballot_sync(FULL_MASK, lane < K && cum > u * tot);
  if (hit) return __ffs(hit) - 1;
  const unsigned pos = __ballot_sync(FULL_MASK, w > 0.f);
  return pos ? 31 - __clz(pos) : 0;
}

// pi_i(rank r) of the proposal law induced by the Select rule.
__device__ __forceinline__ float proposal_mass(const float* ref, int K, int mode, int r) {
  if (mode == BRISK_SELECT_GREEDY) return 1.f;
  float mx = ref[0];
  for (int k = 1; k < K; ++k) mx = fmaxf(mx, ref[k]);
  float tot = 0.f;
  for (int k = 0; k < K; ++k) tot += expf(ref[k] - mx);
  return expf(ref[r] - mx) / tot;
}

// Residual R(v) = max(0, p(v) - pi(v)) of the 8 ids [v0, v0+8) owned by this lane, with
// p(v) = 2^(l(v) log2 e - lse log2 e) on the hardware exponential (v0 is a multiple of 8, so a
// 16-byte-aligned row gives aligned 16-byte vector loads; ragged ends and unaligned rows take
// element loads). Lanes k < K hold candidate k: (cand_id, cand_mass).
__device__ __forceinline__ void residual8(const void* rowp, int dt, int V, float lse, int v0,
                                         int blk0, int cand_id, float cand_mass, int K,
                                         float (&R)[8]) {
  const int lane = threadIdx.x & 31;
  const float nlb = -lse * LOG2E;
  float l[8];
  const bool vec = v0 + 8 <= V && (reinterpret_cast<uintptr_t>(rowp) & 15u) == 0;
  if (vec && dt == BRISK_DT_BF16) {
    unpack(__ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(rowp) + v0)),
           l, __nv_bfloat16());
  } else if (vec) {
    const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const float*>(rowp) + v0);
    float a[4], b[4];
    unpack(__ldg(q), a, 0.f);
    unpack(__ldg(q + 1), b, 0.f);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      l[e] = a[e];
      l[4 + e] = b[e];
    }
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) l[e] = v0 + e < V ? load_logit(rowp, dt, (size_t)(v0 + e)) : -INFINITY;
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) R[e] = ex2(fmaf(l[e], LOG2E, nlb));
  const bool mine = lane < K && cand_id >= blk0 && cand_id < blk0 + RES_BLOCK;
  unsigned mask = __ballot_sync(FULL_MASK, mine);
  while (mask) {
    const int k = __ffs(mask) - 1;
    mask &= mask - 1;
    const int cid = __shfl_sync(FULL_MASK, cand_id, k);
    const float cm = __shfl_sync(FULL_MASK, cand_mass, k);
    const int rel = cid - v0;
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (rel == e) R[e] -= cm;
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) R[e] = fmaxf(R[e], 0.f);
}

// Draw from the normalised [p - pi]_+ of verifier row `rowp` with uniform u, walking ids in
// ascending order; the verifier argmax when the residual mass is <= RESID_Z_FLOOR. CTA-wide.
__device__ int residual_sample(const Smem& sm, const void* rowp, int dt, int V, float lse,
                               const int* cid, const float* ref, int K, int select_mode,
                               int sel_rank, float u, int argmax_p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nblk = (V + RES_BLOCK - 1) / RES_BLOCK;
  // candidate k's proposal mass, held by lane k
  int cand_id = -1;
  float cand_mass = 0.f;
  if (lane < K) {
    cand_id = cid[lane];
    if (select_mode == BRISK_SELECT_GREEDY) cand_mass = (lane == sel_rank) ? 1.f : 0.f;
    else cand_mass = proposal_mass(ref, K, select_mode, lane);
  }
  // pass 1: block sums (blocks interleaved over warps)
  for (int blk = warp; blk < nblk; blk += (int)(blockDim.x >> 5)) {
    const int blk0 = blk * RES_BLOCK;
    float R[8];
    residual8(rowp, dt, V, lse, blk0 + lane * 8, blk0, cand_id, cand_mass, K, R);
    float t = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) t += R[e];
    t = warp_sum(t);
    if (lane == 0) sm.bsum[blk] = t;
  }
  __syncthreads();
  // warp 0: total mass and the block holding the target
  if (warp == 0) {
    const int per = (nblk + 31) / 32;
    const int b0 = lane * per, b1 = min(nblk, b0 + per);
    float mine = 0.f;
    for (int b = b0; b < b1; ++b) mine += sm.bsum[b];
    float incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float o = __shfl_up_sync(FULL_MASK, incl, off);
      if (lane >= off) incl += o;
    }
    const float Z = __shfl_sync(FULL_MASK, incl, 31);
    const float target = u * Z;
    int found = -1;
    float before = 0.f;
    // first lane whose run holds the target, then the block inside the run
    const unsigned hit = __ballot_sync(FULL_MASK, incl > target && b1 > b0);
    if (hit) {
      const int l = __ffs(hit) - 1;
      if (lane == l) {
        float acc = incl - mine;
        for (int b = b0; b < b1; ++b) {
          if (acc + sm.bsum[b] > target) { found = b; break; }
          acc += sm.bsum[b];
        }
        if (found < 0) found = b1 - 1;
        before = acc;
        sm.imisc[0] = found;
        sm.imisc[3] = 0;
        sm.misc[0] = before;
      }
    } else if (lane == 0) {
      // rounding put the target at or past the end: the last id with mass
      int lastb = -1;
      for (int b = nblk - 1; b >= 0; --b)
        if (sm.bsum[b] > 0.f) { lastb = b; break; }
      sm.imisc[0] = lastb;
      sm.imisc[3] = 1;
      sm.misc[0] = 0.f;
    }
    if (lane == 0) {
      sm.misc[1] = Z;
      sm.misc[2] = target;
    }
  }
  __syncthreads();
  const float Z = sm.misc[1];
  if (!(Z > RESID_Z_FLOOR)) return argmax_p;
  const int blk = sm.imisc[0];
  if (blk < 0) return argmax_p;
  // warp 0 walks the block: lane prefix sums, then the lane's 8 ids in order
  if (warp == 0) {
    const int blk0 = blk * RES_BLOCK;
    float R[8];
    residual8(rowp, dt, V, lse, blk0 + lane * 8, blk0, cand_id, cand_mass, K, R);
    float mine = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) mine += R[e];
    float incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float o = __shfl_up_sync(FULL_MASK, incl, off);
      if (lane >= off) incl += o;
    }
    const float before = sm.misc[0];
    const float target = sm.misc[2];
    const bool past_end = sm.imisc[3] != 0;
    const unsigned hit = past_end ? 0u : __ballot_sync(FULL_MASK, before + incl > target);
    int pick = -1;
    if (hit) {
      const int l = __ffs(hit) - 1;
      if (lane == l) {
        float acc = before + incl - mine;
        int lastpos = -1;
        for (int e = 0; e < 8; ++e) {
          if (R[e] > 0.f) lastpos = e;
          acc += R[e];
          if (acc > target) { pick = blk0 + lane * 8 + e; break; }
        }
        if (pick < 0) pick = blk0 + lane * 8 + (lastpos < 0 ? 0 : lastpos);
      }
      pick = __shfl_sync(FULL_MASK, pick, l);
    } else {
      // the last id of the block with positive residual
      const unsigned pos = __ballot_sync(FULL_MASK, mine > 0.f);
      if (pos) {
        const int l = 31 - __clz(pos);
        if (lane == l) {
          int lastpos = 0;
          for (int e = 0; e < 8; ++e)
            if (R[e] > 0.f) lastpos = e;
          pick = blk0 + lane * 8 + lastpos;
        }
        pick = __shfl_sync(FULL_MASK, pick, l);
      } else {
        pick = argmax_p;
      }
    }
    if (lane == 0) sm.imisc[1] = pick;
  }
  __syncthreads();
  return sm.imisc[1];
}

// Left-to-right verification of sm.sel against the verifier rows of sequence b.
__device__ void verify_sequence(const ScanArgs& a, const Smem& sm, int b) {
  const int tid = threadIdx.x;
  const int L = a.L, K = a.K;
  if (tid == 0) sm.imisc[2] = L;
  __syncthreads();
  for (int t = tid; t < L; t += (int)blockDim.x) {
    const size_t bi = (size_t)b * L + t;
    const int x = sm.sel[t];
    bool ok;
    if (a.verify_mode == BRISK_VERIFY_GREEDY) {
      ok = (x == a.argmax_p[bi]);
    } else {
      const float lpx = load_logit(a.logits_p, a.logits_dt, bi * a.V + x);
      const float px = expf(lpx - a.lse_p[bi]);
      const float pim = proposal_mass(sm.ref + (size_t)t * K, K, a.select_mode, sm.rank[t]);
      const float alpha = fminf(1.f, px / pim);
      ok = a.u_acc[bi] < alpha;
    }
    if (!ok) atomicMin(&sm.imisc[2], t);
  }
  __syncthreads();
  const int j = sm.imisc[2];
  int corr = -1;
  if (j < L) {
    const size_t bj = (size_t)b * L + j;
    if (a.verify_mode == BRISK_VERIFY_GREEDY) {
      corr = a.argmax_p[bj];
    } else {
      const void* rowp = (a.logits_dt == BRISK_DT_BF16)
                             ? (const void*)(reinterpret_cast<const __nv_bfloat16*>(a.logits_p) + bj * a.V)
                             : (const void*)(reinterpret_cast<const float*>(a.logits_p) + bj * a.V);
      corr = residual_sample(sm, rowp, a.logits_dt, a.V, a.lse_p[bj], sm.cid + (size_t)j * K,
                             sm.ref + (size_t)j * K, K, a.select_mode, sm.rank[j], a.u_res[bj],
                             a.argmax_p[bj]);
    }
  }
  if (tid == 0) {
    a.accepted_len[b] = j;
    a.correction[b] = (j < L) ? corr : -1;
    if (a.next_anchor) a.next_anchor[b] = (j < L) ? corr : sm.sel[L - 1];
  }
  for (int t = tid; t < L; t += (int)blockDim.x)
    a.out_tokens[(size_t)b * L + t] = t < j ? sm.sel[t] : (t == j ? corr : -1);
}

// Verification of one sequence per CTA (Sec. 3.1; Sec. 3.3; App. B Eq. 6), reading the
// selections and refined scores the corrector wrote.
__global__ void __launch_bounds__(VERIFY_THREADS_MAX)
verify_kernel(const __grid_constant__ ScanArgs a) {
  extern __shared__ __align__(16) char smem_raw[];
  Smem sm;
  smem_layout(a.L, a.K, a.S, a.V, smem_raw, &sm);
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  const int L = a.L, K = a.K, V = a.V;
  const size_t bL = (size_t)b * L;
  // Ids are gathered with below, so out-of-range ones (a row with no finite logit leaves
  // placeholder ids; caller-provided ids may be anything) are replaced by 0 and reported.
  const int nt = (int)blockDim.x;
  for (int e = tid; e < L * K; e += nt) {
    int c = a.cand_ids[bL * K + e];
    if (c < 0 || c >= V) { set_status(a.status, BRISK_ERR_NUMERIC); c = 0; }
    sm.cid[e] = c;
    sm.ref[e] = a.refined[bL * K + e];
  }
  for (int e = tid; e < L; e += nt) {
    int x = a.sel_tokens[bL + e];
    if (x < 0 || x >= V) { set_status(a.status, BRISK_ERR_INVALID_ARG); x = 0; }
    sm.sel[e] = x;
  }
  __syncthreads();
  // each selection's rank in its candidate list
  for (int i = tid; i < L; i += nt) {
    int r = 0;
    for (int k = 0; k < K; ++k)
      if (sm.cid[i * K + k] == sm.sel[i]) { r = k; break; }
    sm.rank[i] = r;
  }
  __syncthreads();
  verify_sequence(a, sm, b);
}

// ---------------------------------------------------------------- corrector
constexpr int CORR_WARPS = 4;   // warps per sequence: one per SM sub-partition

struct CorrSmem {
  float* F;      // [2][S][5]  Fz then Fh
  float* wg;     // [S]
  int* cid;      // [L][K]
  float* clp;    // [L][K]
  float* top;    // [L][3]  l_i(c_0), l_i(c_1), l_i(c_3)
  float* lprev;  // [L][K]  l_i(c_{i-1,k}); row 0 holds l_0(x0) in slot 0
  float* red;    // [2][NW][32] per-warp reduced residual dots (NW > 1)
  float* gpart;  // [2][NW]
  Smem v;        // selections, ranks and refined scores kept for verification in the same CTA
};

__host__ __device__ inline size_t corr_layout(int L, int K, int S, int NW, int V, bool verify,
                                              char* base, CorrSmem* sm) {
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align16(off + bytes);
    return base ? base + o : nullptr;
  };
  char* pF = take(sizeof(float) * 10 * S);
  char* pw = take(sizeof(float) * S);
  char* pc = take(sizeof(int) * L * K);
  char* pl = take(sizeof(float) * L * K);
  char* pt = take(sizeof(float) * L * 3);
  char* pp = take(sizeof(float) * L * K);
  char* pr = take(sizeof(float) * 2 * NW * 32);
  char* pg = take(sizeof(float) * 2 * NW);
  const size_t voff = off;
  if (sm) {
    sm->F = (float*)pF; sm->wg = (float*)pw;
    sm->cid = (int*)pc; sm->clp = (float*)pl; sm->top = (float*)pt; sm->lprev = (float*)pp;
    sm->red = (float*)pr; sm->gpart = (float*)pg;
  }
  // with verification in the same CTA its tables follow (the candidate table is the corrector's)
  if (!verify) return off;
  Smem v;
  off = voff + smem_layout(L, K, S, V, base ? base + voff : nullptr, sm ? &v : nullptr);
  if (sm) {
    sm->v = v;
    sm->v.cid = sm->cid;
  }
  return off;
}

// Warp reduce-scatter of NP values per lane (NP = 8, 16 or 32): afterwards lane l holds the
// warp-wide sum of value (l >> log2(32 / NP)) & (NP - 1), that is value k sits in lane
// k * (32 / NP).
template <int NP>
__device__ __forceinline__ float reduce_scatter_n(float (&v)[NP]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int m = 16, n = NP; n > 1; m >>= 1, n >>= 1) {
    const bool upper = (lane & m) != 0;
#pragma unroll
    for (int j = 0; j < n / 2; ++j) {
      const float send = upper ? v[j] : v[j + n / 2];
      const float keep = upper ? v[j + n / 2] : v[j];
      v[j] = keep + __shfl_xor_sync(FULL_MASK, send, m);
    }
  }
  float r = v[0];
#pragma unroll
  for (int m = 32 / NP / 2; m >= 1; m >>= 1) r += __shfl_xor_sync(FULL_MASK, r, m);
  return r;
}

// Gathers n logits, entry e at index_of(e) into *dst_of(e), eight loads in flight per lane.
template <int NT, typename IndexOf, typename DstOf>
__device__ __forceinline__ void gather_logits(const void* logits, int dt, int n, IndexOf index_of,
                                              DstOf dst_of) {
  const int tid = threadIdx.x;
  for (int base = 0; base < n; base += 8 * NT) {
    float v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int e = base + j * NT + tid;
      v[j] = e < n ? load_logit(logits, dt, index_of(e)) : 0.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int e = base + j * NT + tid;
      if (e < n) *dst_of(e) = v[j];
    }
  }
}

// The sequential corrector (Sec. 3.3 Eqs. 4-5; App. C.3 Eq. 9; Algorithm 1(b) loop), one CTA of
// NW warps per sequence. Lane l of warp w owns the CW-element state chunks (CW = 1, 2 or 4)
// c = l + 32 (w + NW m), m < CMC. The residual dots and the gate are reduced with warp
// shuffles, then across the warps through shared memory (one block barrier a position), and
// Select runs in every warp with lane k holding candidate k. Spreading a sequence over the
// SM's four sub-partitions shortens the dependent chain of a position and keeps each
// sub-partition's share small, so the verifier-row sweep beside it keeps its issue slots.
// Every load of the step is issued unconditionally (chunk and candidate indices clamped into
// range, the surplus contributions multiplied by zero state or never read) so the compiler can
// keep them all in flight. Table rows are read through L2 (cache-global loads) a whole position
// ahead into registers; an L2 line prefetch two positions ahead on top of that was slower
// (single 105.7 -> 102.5 us for the products and the corrector without it, large_vocab
// 269 -> 253 us). Shared memory holds the per-sequence tables (candidates, their log-probs, the
// features' logits) and, for 4-element chunks, the feature shares and gate weights.
// VERIFY: the CTA also verifies its sequence after the scan (the fused small-batch schedule); a
// separate instantiation, since the verification code raises the scan's register count (122 ->
// 143 a thread for four warps of 2-element chunks and K = 8), which would leave less room for
// the verifier-row sweep beside the corrector in the overlapping schedule.
template <int NW, int NP, int CMC, int CW, bool VERIFY>
__global__ void __launch_bounds__(NW * 32)
corrector_kernel(const __grid_constant__ ScanArgs a) {
  extern __shared__ __align__(16) char smem_raw[];
  CorrSmem sm;
  corr_layout(a.L, a.K, a.S, NW, a.V, VERIFY, smem_raw, &sm);
  constexpr int NT = NW * 32;
  constexpr int LSTEP = 32 / NP;           // lane stride between reduced dots
  const int b = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int L = a.L, K = a.K, S = a.S, V = a.V;
  const size_t bL = (size_t)b * L;
  const int nch = S / CW;

  // Prologue in two dependent rounds of loads. First everything that depends neither on the
  // candidates nor on x0, issued at once with the candidate table itself; then, after one
  // barrier, what depends on them (the token shares of x0, the first position's residual rows
  // and the features' logit gathers, in one batch).
  // lane chunks, clamped into range; a chunk past the state keeps s = 0 throughout
  int cc[CMC];
  bool ok[CMC];
#pragma unroll
  for (int m = 0; m < CMC; ++m) {
    const int c = lane + 32 * (warp + NW * m);
    ok[m] = c < nch;
    cc[m] = ok[m] ? c : nch - 1;
  }
  using C = Chunk<CW>;
  int x0 = a.x0[b];
  // the Init share of h_c and the first position's hidden and position shares
  C g0c[CMC], gz4[CMC], gh4[CMC], pz0[CMC], ph0[CMC];
#pragma unroll
  for (int m = 0; m < CMC; ++m) {
    const int c = cc[m];
    g0c[m] = ldc<CW, true>(a.G0 + (size_t)b * S + CW * c);
    gz4[m] = ldc<CW, true>(a.G + bL * 2 * S + CW * c);
    gh4[m] = ldc<CW, true>(a.G + bL * 2 * S + S + CW * c);
    pz0[m] = ldc<CW, false>(a.posG + CW * c);
    ph0[m] = ldc<CW, false>(a.posG + S + CW * c);
  }
  float wgf[5];
#pragma unroll
  for (int f = 0; f < 5; ++f) wgf[f] = a.wg[S + f];
  // chunks of up to two elements: this lane's feature shares (5 CW floats of F[S, 5] for z and
  // for h) and gate weights, read every step, held in registers for the whole scan (4-element
  // chunks read them from shared memory: in registers they would spill)
  constexpr bool FREG = CW <= 2;
  constexpr int FR = FREG ? CMC : 1;
  float fzr[FR][5 * CW], fhr[FR][5 * CW];
  C wgr[FR];
  if constexpr (FREG) {
#pragma unroll
    for (int m = 0; m < CMC; ++m) {
#pragma unroll
      for (int q = 0; q < 5; ++q) {
        const C vz = ldc<CW, false>(a.Fz + 5 * CW * cc[m] + CW * q);
        const C vh = ldc<CW, false>(a.Fh + 5 * CW * cc[m] + CW * q);
#pragma unroll
        for (int e = 0; e < CW; ++e) {
          fzr[m][CW * q + e] = vz.v[e];
          fhr[m][CW * q + e] = vh.v[e];
        }
      }
      wgr[m] = ldc<CW, false>(a.wg + CW * cc[m]);
    }
  }
  const float sig_alpha = sigmoidf_(a.alpha);
  // the candidate table
  for (int e = tid; e < L * K; e += NT) {
    int c = a.cand_ids[bL * K + e];
    if (c < 0 || c >= V) { set_status(a.status, BRISK_ERR_NUMERIC); c = 0; }
    sm.cid[e] = c;
    sm.clp[e] = a.cand_logprob[bL * K + e];
  }
  if (x0 < 0 || x0 >= V) {
    if (tid == 0) set_status(a.status, BRISK_ERR_INVALID_ARG);
    x0 = 0;
  }
  if constexpr (!FREG) {
    // the feature shares and the gate weights into shared memory, all loads first
    constexpr int FV = 2 * 5 * 1024 / 4 / NT + 1;   // float4 of Fz and Fh a thread, S <= 1024
    float4 fv[FV];
    const int nf = 5 * S / 4;
#pragma unroll
    for (int j = 0; j < FV; ++j) {
      const int e = tid + j * NT;
      fv[j] = e < nf ? ld4(a.Fz + 4 * e) : (e < 2 * nf ? ld4(a.Fh + 4 * (e - nf)) : float4{});
    }
    const float4 wv = tid < S / 4 ? ld4(a.wg + 4 * tid) : float4{};
#pragma unroll
    for (int j = 0; j < FV; ++j) {
      const int e = tid + j * NT;
      if (e < 2 * nf) reinterpret_cast<float4*>(sm.F)[e] = fv[j];
    }
    for (int e = tid; e < S / 4; e += NT)
      reinterpret_cast<float4*>(sm.wg)[e] = e == tid ? wv : ld4(a.wg + 4 * e);
  }
  __syncthreads();

  // second round: the token shares of x0, the first position's residual rows (below) and the
  // features' logit gathers, all independent of the selections
  C t0c[CMC], tz4[CMC], th4[CMC];
#pragma unroll
  for (int m = 0; m < CMC; ++m) {
    const int c = cc[m];
    t0c[m] = ldc<CW, true>(a.T0 + (size_t)x0 * S + CW * c);
    tz4[m] = ldc<CW, true>(a.Tzh + (size_t)x0 * 2 * S + CW * c);   // token share of x_{-1} = x0
    th4[m] = ldc<CW, true>(a.Tzh + (size_t)x0 * 2 * S + S + CW * c);
  }
  const void* lq = a.logits_q;
  const int ldt = a.logits_dt;
  gather_logits<NT>(
      lq, ldt, L * 3 + L * K,
      [&](int e) {
        if (e < L * 3) {
          const int i = e / 3, w = e % 3;
          return (bL + i) * V + sm.cid[i * K + (w == 0 ? 0 : (w == 1 ? 1 : 3))];
        }
        e -= L * 3;
        const int i = e / K, k = e % K;
        return i == 0 ? bL * V + x0 : (bL + i) * V + sm.cid[(i - 1) * K + k];
      },
      [&](int e) { return e < L * 3 ? sm.top + e : sm.lprev + (e - L * 3); });
  C s4[CMC];
#pragma unroll
  for (int m = 0; m < CMC; ++m) {
#pragma unroll
    for (int e = 0; e < CW; ++e)                              // s_{-1} = u_0 = Init(h_c, E(x0))
      s4[m].v[e] = ok[m] ? tanhf(g0c[m].v[e] + t0c[m].v[e]) : 0.f;
    gz4[m] = addc(gz4[m], pz0[m]);
    gh4[m] = addc(gh4[m], ph0[m]);
  }
  __syncthreads();

  // Software pipeline across positions: the next position's residual rows (rank K-1 repeated
  // past K) and hidden and position shares are loaded into registers one step ahead (issued at
  // the top of the step: issued after the step's dots they were still in flight when the next
  // step began, single 118 -> 110 us for the products and the corrector), and so is the
  // token-share row of this position's rank-0 candidate, the usual next previous token.
  // (Only while the rows fit in registers: NP * CMC <= 16 vectors a lane; wider variants load
  // them in the step.)
  constexpr bool PIPE = NP * CMC <= 16;
  constexpr int PK = PIPE ? NP : 1;
  C ub[PK][CMC];
  if constexpr (PIPE) {
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      const float* Uk = a.U + (size_t)sm.cid[k < K ? k : K - 1] * S;
#pragma unroll
      for (int m = 0; m < CMC; ++m) ub[k][m] = ldc<CW, true>(Uk + CW * cc[m]);
    }
  }
  C tsz[CMC], tsh[CMC];                      // token share of the speculated previous token
  int ts_id = -1;

  int prev = x0, prank = 0;
  float u_cur = (a.select_mode == BRISK_SELECT_SAMPLE) ? a.u_sel[bL] : 0.f;
  for (int i = 0; i < L; ++i) {
    const int buf = i & 1;
    const int* ci = sm.cid + i * K;
    // into registers, for step i + 1: its hidden and position shares, residual rows and the
    // rank-0 token-share row
    C un[PK][CMC], tnz[CMC], tnh[CMC], gnz[CMC], gnh[CMC], pnz[CMC], pnh[CMC];
    if (i + 1 < L) {
      const float* Gn = a.G + (bL + i + 1) * 2 * S;
      const float* Pn = a.posG + (size_t)(i + 1) * 2 * S;
#pragma unroll
      for (int m = 0; m < CMC; ++m) {
        gnz[m] = ldc<CW, true>(Gn + CW * cc[m]);
        gnh[m] = ldc<CW, true>(Gn + S + CW * cc[m]);
        pnz[m] = ldc<CW, false>(Pn + CW * cc[m]);
        pnh[m] = ldc<CW, false>(Pn + S + CW * cc[m]);
      }
      if constexpr (PIPE) {
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          const float* Uk = a.U + (size_t)ci[K + (k < K ? k : K - 1)] * S;
#pragma unroll
          for (int m = 0; m < CMC; ++m) un[k][m] = ldc<CW, true>(Uk + CW * cc[m]);
        }
      }
      const float* Tn = a.Tzh + (size_t)ci[0] * 2 * S;
#pragma unroll
      for (int m = 0; m < CMC; ++m) {
        tnz[m] = ldc<CW, true>(Tn + CW * cc[m]);
        tnh[m] = ldc<CW, true>(Tn + S + CW * cc[m]);
      }
    }
    // confidence features of position i (App. C.3)
    const float l0 = sm.top[i * 3 + 0];
    float phi[5];
    phi[0] = l0 - sm.top[i * 3 + 1];
    phi[1] = l0 - sm.top[i * 3 + 2];
    phi[2] = (prev == ci[0]) ? 1.f : 0.f;
    phi[3] = (prev == ci[0] || prev == ci[1] || prev == ci[2] || prev == ci[3]) ? 1.f : 0.f;
    phi[4] = l0 - sm.lprev[i * K + (i == 0 ? 0 : prank)];
    // token share of the previous token (x0's came with the prologue; the speculated one is
    // already in registers)
    if (i > 0) {
      if (prev == ts_id) {
#pragma unroll
        for (int m = 0; m < CMC; ++m) {
          tz4[m] = tsz[m];
          th4[m] = tsh[m];
        }
      } else {
        const float* Tp = a.Tzh + (size_t)prev * 2 * S;
#pragma unroll
        for (int m = 0; m < CMC; ++m) {
          tz4[m] = ldc<CW, true>(Tp + CW * cc[m]);
          th4[m] = ldc<CW, true>(Tp + S + CW * cc[m]);
        }
      }
    }
    // minimal-GRU step on this lane's chunks and its gate partial
    float gacc = 0.f;
#pragma unroll
    for (int m = 0; m < CMC; ++m) {
      const int c = cc[m];
      C zp = addc(gz4[m], tz4[m]), hp = addc(gh4[m], th4[m]);
      // feature shares of this chunk's elements: 5 CW contiguous floats of F[S, 5]
      float fz[5 * CW], fh[5 * CW];
      if constexpr (FREG) {
#pragma unroll
        for (int j = 0; j < 5 * CW; ++j) {
          fz[j] = fzr[m][j];
          fh[j] = fhr[m][j];
        }
      } else {
#pragma unroll
        for (int q = 0; q < 5; ++q) {
          const C vz = ldc<CW, false>(sm.F + 5 * CW * c + CW * q);
          const C vh = ldc<CW, false>(sm.F + 5 * S + 5 * CW * c + CW * q);
#pragma unroll
          for (int e = 0; e < CW; ++e) {
            fz[CW * q + e] = vz.v[e];
            fh[CW * q + e] = vh.v[e];
          }
        }
      }
#pragma unroll
      for (int e = 0; e < CW; ++e)
#pragma unroll
        for (int f = 0; f < 5; ++f) {
          zp.v[e] = fmaf(fz[5 * e + f], phi[f], zp.v[e]);
          hp.v[e] = fmaf(fh[5 * e + f], phi[f], hp.v[e]);
        }
#pragma unroll
      for (int e = 0; e < CW; ++e) {
        const float z = sigmoid_fast(zp.v[e]);
        s4[m].v[e] = ok[m] ? (1.f - z) * s4[m].v[e] + z * hp.v[e] : 0.f;
      }
      if constexpr (FREG) gacc = dotc(wgr[m], s4[m], gacc);
      else gacc = dotc(ldc<CW, false>(sm.wg + CW * c), s4[m], gacc);
    }
    // residual-dot partials with the rows of this position's candidates
    float part[NP];
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      const float* Uk = a.U + (size_t)ci[k < K ? k : K - 1] * S;
      float acc = 0.f;
#pragma unroll
      for (int m = 0; m < CMC; ++m) {
        C u;
        if constexpr (PIPE) u = ub[k][m];
        else u = ldc<CW, true>(Uk + CW * cc[m]);
        acc = dotc(u, s4[m], acc);
      }
      part[k] = acc;
    }
    // hidden and position shares of the next position: plain loads first used in the next step
    if (i + 1 < L) {
#pragma unroll
      for (int m = 0; m < CMC; ++m) {
        gz4[m] = addc(gnz[m], pnz[m]);
        gh4[m] = addc(gnh[m], pnh[m]);
      }
    }
    // residual dots by a warp reduce-scatter; across warps through shared memory, where lane k
    // sums the warps' partials of dot k (one shuffle fewer on the step's chain than summing in
    // the reduce-scatter's lanes and moving dot k to lane k afterwards)
    const float r = reduce_scatter_n<NP>(part);
    gacc = warp_sum(gacc);
    float dk;
    if constexpr (NW > 1) {
      float* red = sm.red + buf * NW * 32;
      if ((lane & (LSTEP - 1)) == 0) red[warp * 32 + lane / LSTEP] = r;
      if (lane == 0) sm.gpart[buf * NW + warp] = gacc;
      __syncthreads();
      const int vidx = lane & (NP - 1);
      dk = red[vidx];
      gacc = sm.gpart[buf * NW];
      for (int w = 1; w < NW; ++w) {
        dk += red[w * 32 + vidx];
        gacc += sm.gpart[buf * NW + w];
      }
    } else {
      dk = __shfl_sync(FULL_MASK, r, (lane * LSTEP) & 31);
    }
    // gate, refined scores (lane k: candidate k) and Select, identically in every warp
    float gate = a.b_g + gacc;
#pragma unroll
    for (int f = 0; f < 5; ++f) gate = fmaf(wgf[f], phi[f], gate);
    const float gamma = sig_alpha * sigmoid_fast(gate);
    const float ref = lane < K ? sm.clp[i * K + lane] + gamma * dk : -INFINITY;
    const float u_cur_draw = u_cur;
    const int pick = select_warp(ref, K, a.select_mode, u_cur);
    if (warp == 0) {
      if (lane < K) a.refined[(bL + i) * K + lane] = ref;
      if (__any_sync(FULL_MASK, lane < K && isnan(ref)) && lane == 0)
        set_status(a.status, BRISK_ERR_NUMERIC);
    }
    if (a.select_mode == BRISK_SELECT_SAMPLE && i + 1 < L) u_cur = a.u_sel[bL + i + 1];
    if (tid == 0) {
      a.sel_tokens[bL + i] = ci[pick];
      if constexpr (VERIFY) {
        sm.v.sel[i] = ci[pick];
        sm.v.rank[i] = pick;
      }
    }
    if constexpr (VERIFY)
      if (warp == 0 && lane < K) sm.v.ref[i * K + lane] = ref;
    // the token fed forward: the head's selection, or in a same-state replay the base
    // selection (the Select rule on the base scores log q, same draw)
    int fwd = pick;
    if (a.base_prefix) {
      fwd = select_warp(lane < K ? sm.clp[i * K + lane] : -INFINITY, K, a.select_mode, u_cur_draw);
      if (tid == 0) a.base_rank[bL + i] = fwd;
    }
    prank = fwd;
    prev = ci[fwd];
    // advance the pipeline
    if (i + 1 < L) {
      if constexpr (PIPE) {
#pragma unroll
        for (int k = 0; k < NP; ++k)
#pragma unroll
          for (int m = 0; m < CMC; ++m) ub[k][m] = un[k][m];
      }
#pragma unroll
      for (int m = 0; m < CMC; ++m) {
        tsz[m] = tnz[m];
        tsh[m] = tnh[m];
      }
      ts_id = ci[0];
    }
  }
  // verification of this sequence in the same CTA (the verifier rows' statistics are complete:
  // their sweep ran before this kernel)
  if constexpr (VERIFY) {
    __syncthreads();
    verify_sequence(a, sm.v, b);
  }
}

}  // namespace

size_t scan_smem_bytes(int L, int K, int S, int V) {
  return smem_layout(L, K, S, V, nullptr, nullptr);
}

template <int NW, int NP, int CMC, int CW, bool VERIFY>
cudaError_t launch_corrector_k(const ScanArgs& a, cudaStream_t stream) {
  const size_t smem = corr_layout(a.L, a.K, a.S, NW, a.V, VERIFY, nullptr, nullptr);
  auto kernel = corrector_kernel<NW, NP, CMC, CW, VERIFY>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = prefer_carveout(kernel, CARVEOUT_SMALL_KB);
  if (e != cudaSuccess) return e;
  e = launch_prio(kernel, dim3(a.B), dim3(NW * 32), smem, stream, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int NW, int CW, int NP>
cudaError_t launch_corrector(const ScanArgs& a, cudaStream_t stream) {
  if (a.do_verify) return launch_corrector_k<NW, NP, 1, CW, true>(a, stream);
  return launch_corrector_k<NW, NP, 1, CW, false>(a, stream);
}

template <int NW, int CW>
cudaError_t launch_corrector_for_k(const ScanArgs& a, cudaStream_t stream) {
  if (a.K <= 8) return launch_corrector<NW, CW, 8>(a, stream);
  return a.K <= 16 ? launch_corrector<NW, CW, 16>(a, stream) : launch_corrector<NW, CW, 32>(a, stream);
}

// The corrector (do_select; with do_verify also the verification in the same CTA) or the
// verification alone (do_verify) for every sequence.
cudaError_t launch_scan(const ScanArgs& a, cudaStream_t stream) {
  if (a.do_select) {
    // One chunk a lane. A state of up to 256 takes four warps, one per SM sub-partition, of
    // 1- or 2-element chunks (every lane busy); 257..512 eight warps of 2-element chunks and a
    // wider one (up to 1024) eight warps of 4-element chunks: two warps of the sequence on each
    // sub-partition to issue from. (At S = 512 eight warps of 2-element chunks beat four of
    // 4-element chunks, single 144 -> 135 us a tail, and sixteen of single elements, 138 us:
    // the cross-warp sums grow with the warps.)
    if (a.S > 4 * 32 * CORR_WARPS) return launch_corrector_for_k<2 * CORR_WARPS, 4>(a, stream);
    if (a.S > 2 * 32 * CORR_WARPS) return launch_corrector_for_k<2 * CORR_WARPS, 2>(a, stream);
    if (a.S > 32 * CORR_WARPS) return launch_corrector_for_k<CORR_WARPS, 2>(a, stream);
    return launch_corrector_for_k<CORR_WARPS, 1>(a, stream);
  }
  const size_t smem = scan_smem_bytes(a.L, a.K, a.S, a.V);
  cudaError_t e = cudaFuncSetAttribute(verify_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e == cudaSuccess) e = prefer_carveout(verify_kernel, CARVEOUT_SMALL_KB);
  if (e != cudaSuccess) return e;
  const int threads = a.verify_mode == BRISK_VERIFY_STOCHASTIC ? VERIFY_THREADS_MAX : VERIFY_THREADS;
  e = launch_prio(verify_kernel, dim3(a.B), dim3(threads), smem, stream, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace brisk
