// Corrector scan and verification, one CTA per sequence.
//
// Corrector (Sec. 3.3 Eqs. 4-5; App. C.2 Eq. 7; Algorithm 1(b) loop). The
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
// Verification (Sec. 3.1; Sec. 3.3; App. B Eq. 8) runs in the same CTA after
// the scan, or alone (brisk_verify_block), through the same device code.
#include "brisk_internal.cuh"

namespace brisk {

namespace {

constexpr int SCAN_THREADS = 128;
constexpr int SCAN_WARPS = SCAN_THREADS / 32;
constexpr int MCH = 2;          // 4-element state chunks per thread: S <= 4 * 128 * MCH = 1024

struct Smem {
  float* s;        // [S]     state (read back by nothing in the step loop; kept for debugging layout)
  float* F;        // [10][S] Fz then Fh, feature-major
  float* gpart;    // [2][SCAN_WARPS] gate partial sums (double-buffered)
  float* red;      // [2][SCAN_WARPS][32] residual-dot partial sums after the warp reduce-scatter
  int* cid;        // [L][K]
  float* clp;      // [L][K]
  float* top;      // [L][3]  l_i(c_0), l_i(c_1), l_i(c_3)
  float* lprev;    // [L][K]  l_i(c_{i-1,k}); row 0 holds l_0(x0) in slot 0
  int* sel;        // [L]
  int* rank;       // [L]
  float* ref;      // [L][K]
  float* bsum;     // [nblk]  residual block sums
  float* misc;     // [16]
  int* imisc;      // [16]
  float* U;        // [nbuf][K][S]  residual rows of a position's candidates
  float* Tc;       // [nbuf][K][2S] token-share rows of the previous position's candidates
  uint64_t* full;  // [nbuf] mbarriers: the bulk copies of a buffer have landed
};

__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

constexpr int RES_BLOCK = 256;  // residual-sampling block: 32 lanes x 8 ids

__host__ __device__ inline size_t smem_layout(int L, int K, int S, int V, int nbuf, int tcand,
                                              char* base, Smem* sm) {
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align16(off + bytes);
    return base ? base + o : nullptr;
  };
  const int nblk = (V + RES_BLOCK - 1) / RES_BLOCK;
  char* p_s = take(sizeof(float) * S);
  char* p_F = take(sizeof(float) * 10 * S);
  char* p_g = take(sizeof(float) * 2 * SCAN_WARPS);
  char* p_red = take(sizeof(float) * 2 * SCAN_WARPS * 32);
  char* p_cid = take(sizeof(int) * L * K);
  char* p_clp = take(sizeof(float) * L * K);
  char* p_top = take(sizeof(float) * L * 3);
  char* p_lprev = take(sizeof(float) * L * K);
  char* p_sel = take(sizeof(int) * L);
  char* p_rank = take(sizeof(int) * L);
  char* p_ref = take(sizeof(float) * L * K);
  char* p_bsum = take(sizeof(float) * nblk);
  char* p_misc = take(sizeof(float) * 16);
  char* p_imisc = take(sizeof(int) * 16);
  char* p_U = take(sizeof(float) * nbuf * K * S);
  char* p_Tc = take(tcand ? sizeof(float) * nbuf * K * 2 * S : 0);
  char* p_full = take(sizeof(uint64_t) * 4);
  if (sm) {
    sm->full = (uint64_t*)p_full;
    sm->s = (float*)p_s; sm->F = (float*)p_F; sm->gpart = (float*)p_g; sm->red = (float*)p_red;
    sm->cid = (int*)p_cid; sm->clp = (float*)p_clp; sm->top = (float*)p_top;
    sm->lprev = (float*)p_lprev; sm->sel = (int*)p_sel; sm->rank = (int*)p_rank;
    sm->ref = (float*)p_ref; sm->bsum = (float*)p_bsum; sm->misc = (float*)p_misc;
    sm->imisc = (int*)p_imisc; sm->U = (float*)p_U; sm->Tc = (float*)p_Tc;
  }
  return off;
}

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
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
constexpr long long SCAN_WAIT_LIMIT_CYCLES = 4000000000ll;   // about 2 s of SM clock
// Bounded wait for a phase of an mbarrier; false when it expired.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (unsigned n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 63) == 0 && clock64() - t0 > SCAN_WAIT_LIMIT_CYCLES) return false;
  }
}
// Bulk (TMA) copy of `bytes` (a multiple of 16, 16-byte aligned ends) completing on `bar`.
__device__ __forceinline__ void bulk_copy(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          su32(dst)),
      "l"(src), "r"(bytes), "r"(su32(bar))
      : "memory");
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

// Residual dot d_k of one position: the four warps' partial sums, added in a fixed order.
__device__ __forceinline__ float dot_k(const float* red, int k) {
  return ((red[k] + red[32 + k]) + red[64 + k]) + red[96 + k];
}

// Select with lane k holding refined score k (lanes >= K hold -inf); the same in every lane.
// Greedy: argmax, the lowest rank on ties. Sample: the first rank whose cumulative softmax mass
// exceeds u * total (warp prefix sums), else the last rank with mass.
__device__ __forceinline__ int select_warp(float ref, int K, int mode, float u) {
  const int lane = threadIdx.x & 31;
  if (mode == BRISK_SELECT_GREEDY) {
    float bv = ref;
    int bk = lane < K ? lane : 0x7fffffff;
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      const float ov = __shfl_xor_sync(FULL_MASK, bv, off);
      const int ok = __shfl_xor_sync(FULL_MASK, bk, off);
      if (ov > bv || (ov == bv && ok < bk)) { bv = ov; bk = ok; }
    }
    return bk;
  }
  const float mx = warp_max(ref);
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

// Residual R(v) = max(0, p(v) - pi(v)) of the 8 ids [v0, v0+8) owned by this lane.
// Lanes k < K hold candidate k: (cand_id, cand_mass).
__device__ __forceinline__ void residual8(const void* rowp, int dt, int V, float lse, int v0,
                                         int blk0, int cand_id, float cand_mass, int K,
                                         float (&R)[8]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int v = v0 + e;
    R[e] = (v < V) ? expf(load_logit(rowp, dt, (size_t)v) - lse) : 0.f;
  }
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
  for (int blk = warp; blk < nblk; blk += SCAN_WARPS) {
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
  for (int t = tid; t < L; t += SCAN_THREADS) {
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
  for (int t = tid; t < L; t += SCAN_THREADS)
    a.out_tokens[(size_t)b * L + t] = t < j ? sm.sel[t] : (t == j ? corr : -1);
}

// The sequential corrector over the positions of sequence b (Algorithm 1(b) loop). Thread t owns
// the 4-element state chunks c = t + 128 m: it updates them, stages its own chunks of the
// candidates' residual and token-share rows with cp.async (nbuf - 1 positions ahead; no other
// thread reads them, so its own wait suffices), and contributes its partial residual dots, which
// one warp reduce-scatter and one block barrier per position turn into the K dots.
template <int NP>
__device__ void corrector_loop(const ScanArgs& a, const Smem& sm, int b, int x0) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int L = a.L, K = a.K, S = a.S;
  const size_t bL = (size_t)b * L;
  const int nch = S / 4;
  const int nbuf = a.ubuf, tcand = a.tcand;

  float4 s4[MCH], wg4[MCH], gz4[MCH], gh4[MCH], tz4[MCH], th4[MCH];
#pragma unroll
  for (int m = 0; m < MCH; ++m) {
    const int c = tid + m * SCAN_THREADS;
    s4[m] = wg4[m] = gz4[m] = gh4[m] = tz4[m] = th4[m] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c < nch) {
      const float4 g0 = ld4(a.G0 + (size_t)b * S + 4 * c), t0 = ld4(a.T0 + (size_t)x0 * S + 4 * c);
      s4[m] = make_float4(tanhf(g0.x + t0.x), tanhf(g0.y + t0.y), tanhf(g0.z + t0.z),
                          tanhf(g0.w + t0.w));                     // s_{-1} = u_0 = Init(h_c, E(x0))
      wg4[m] = ld4(a.wg + 4 * c);
      gz4[m] = ld4(a.G + bL * 2 * S + 4 * c);
      gh4[m] = ld4(a.G + bL * 2 * S + S + 4 * c);
      tz4[m] = ld4(a.Tzh + (size_t)x0 * 2 * S + 4 * c);           // token share of x_{-1} = x0
      th4[m] = ld4(a.Tzh + (size_t)x0 * 2 * S + S + 4 * c);
    }
  }
  float wgf[5];
#pragma unroll
  for (int f = 0; f < 5; ++f) wgf[f] = a.wg[S + f];
  const float sig_alpha = sigmoidf_(a.alpha);

  // The rows position j needs (the residual rows of its candidates and, when staged, the
  // token-share rows of the previous position's candidates) arrive in buffer j % nbuf by bulk
  // copies that thread 0 issues; everybody waits on that buffer's mbarrier.
  const uint32_t u_bytes = (uint32_t)S * 4, t_bytes = (uint32_t)S * 8;
  auto issue = [&](int j) {
    if (tid != 0 || j >= L) return;
    const int slot = j % nbuf;
    float* Ub = sm.U + (size_t)slot * K * S;
    float* Tb = sm.Tc + (size_t)slot * K * 2 * S;
    const bool with_t = tcand && j > 0;
    mbar_expect_tx(&sm.full[slot], K * (u_bytes + (with_t ? t_bytes : 0)));
    for (int k = 0; k < K; ++k) {
      bulk_copy(Ub + (size_t)k * S, a.U + (size_t)sm.cid[j * K + k] * S, u_bytes, &sm.full[slot]);
      if (with_t)
        bulk_copy(Tb + (size_t)k * 2 * S, a.Tzh + (size_t)sm.cid[(j - 1) * K + k] * 2 * S, t_bytes,
                  &sm.full[slot]);
    }
  };
  if (tid == 0) {
    for (int q = 0; q < nbuf; ++q) mbar_init(&sm.full[q], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int ahead = nbuf > 1 ? nbuf - 1 : 0;
  for (int j = 0; j < (nbuf > 1 ? ahead : 1); ++j) issue(j);
  // this thread's share of the L2 prefetch of a table row: fixed across positions
  const int u_lines = (S * 4 + 127) / 128, t_lines = (S * 8 + 127) / 128;
  const int pu_k = tid / u_lines, pu_l = tid % u_lines;
  bool timed_out = false;

  int prev = x0, prank = 0;
  float u_cur = (a.select_mode == BRISK_SELECT_SAMPLE) ? a.u_sel[bL] : 0.f;
  for (int i = 0; i < L; ++i) {
    const int buf = i & 1;
    const int* ci = sm.cid + i * K;
    if (nbuf > 1) issue(i + ahead);
    // L2 prefetch further ahead (and of the gathered token-share rows when they are not staged)
    if (i + nbuf < L && pu_k < K) prefetch_l2(a.U + (size_t)ci[nbuf * K + pu_k] * S + pu_l * 32);
    if (!tcand && i + 1 < L)
      for (int e = tid; e < K * t_lines; e += SCAN_THREADS)
        prefetch_l2(a.Tzh + (size_t)ci[e / t_lines] * 2 * S + (e % t_lines) * 32);
    // confidence features of position i (App. C.2)
    const float l0 = sm.top[i * 3 + 0];
    float phi[5];
    phi[0] = l0 - sm.top[i * 3 + 1];
    phi[1] = l0 - sm.top[i * 3 + 2];
    phi[2] = (prev == ci[0]) ? 1.f : 0.f;
    phi[3] = (prev == ci[0] || prev == ci[1] || prev == ci[2] || prev == ci[3]) ? 1.f : 0.f;
    phi[4] = l0 - sm.lprev[i * K + (i == 0 ? 0 : prank)];
    // the rows of position i have landed
    if (!mbar_wait(&sm.full[i % nbuf], (i / nbuf) & 1)) timed_out = true;
    const float* Ub = sm.U + (size_t)(i % nbuf) * K * S;
    // token share of the previous token (x0's came with the prologue)
    if (i > 0) {
      const float* Tp = tcand ? sm.Tc + ((size_t)(i % nbuf) * K + prank) * 2 * S
                              : a.Tzh + (size_t)prev * 2 * S;
#pragma unroll
      for (int m = 0; m < MCH; ++m) {
        const int c = tid + m * SCAN_THREADS;
        if (c < nch) {
          tz4[m] = ld4(Tp + 4 * c);
          th4[m] = ld4(Tp + S + 4 * c);
        }
      }
    }
    // minimal-GRU step on this thread's chunks, its gate partial and its residual-dot partials
    float gacc = 0.f;
    float part[NP];
#pragma unroll
    for (int k = 0; k < NP; ++k) part[k] = 0.f;
#pragma unroll
    for (int m = 0; m < MCH; ++m) {
      const int c = tid + m * SCAN_THREADS;
      if (c < nch) {
        float zp[4] = {gz4[m].x + tz4[m].x, gz4[m].y + tz4[m].y, gz4[m].z + tz4[m].z,
                       gz4[m].w + tz4[m].w};
        float hp[4] = {gh4[m].x + th4[m].x, gh4[m].y + th4[m].y, gh4[m].z + th4[m].z,
                       gh4[m].w + th4[m].w};
#pragma unroll
        for (int f = 0; f < 5; ++f) {
          const float4 fz = ld4(sm.F + (size_t)f * S + 4 * c);
          const float4 fh = ld4(sm.F + (size_t)(5 + f) * S + 4 * c);
          zp[0] = fmaf(fz.x, phi[f], zp[0]); zp[1] = fmaf(fz.y, phi[f], zp[1]);
          zp[2] = fmaf(fz.z, phi[f], zp[2]); zp[3] = fmaf(fz.w, phi[f], zp[3]);
          hp[0] = fmaf(fh.x, phi[f], hp[0]); hp[1] = fmaf(fh.y, phi[f], hp[1]);
          hp[2] = fmaf(fh.z, phi[f], hp[2]); hp[3] = fmaf(fh.w, phi[f], hp[3]);
        }
        float sv[4] = {s4[m].x, s4[m].y, s4[m].z, s4[m].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float z = sigmoid_fast(zp[e]);
          sv[e] = (1.f - z) * sv[e] + z * hp[e];
        }
        s4[m] = make_float4(sv[0], sv[1], sv[2], sv[3]);
        gacc = fmaf(wg4[m].x, sv[0], gacc);
        gacc = fmaf(wg4[m].y, sv[1], gacc);
        gacc = fmaf(wg4[m].z, sv[2], gacc);
        gacc = fmaf(wg4[m].w, sv[3], gacc);
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          if (k < K) {
            const float4 u = ld4(Ub + (size_t)k * S + 4 * c);
            part[k] = fmaf(u.x, sv[0], fmaf(u.y, sv[1], fmaf(u.z, sv[2], fmaf(u.w, sv[3], part[k]))));
          }
        }
      }
    }
    // hidden and position shares of the next position: plain loads first used in the next step
    if (i + 1 < L) {
      const float* Gn = a.G + (bL + i + 1) * 2 * S;
#pragma unroll
      for (int m = 0; m < MCH; ++m) {
        const int c = tid + m * SCAN_THREADS;
        if (c < nch) {
          gz4[m] = ld4(Gn + 4 * c);
          gh4[m] = ld4(Gn + S + 4 * c);
        }
      }
    }
    // block reduction: residual dots by one reduce-scatter per warp, gate partial by a warp sum
    const float r = reduce_scatter<NP>(part);
    const int v = NP == 16 ? ((lane >> 1) & 15) : lane;
    float* red = sm.red + buf * SCAN_WARPS * 32;
    if (v < K && (NP == 32 || (lane & 1) == 0)) red[warp * 32 + v] = r;
    gacc = warp_sum(gacc);
    if (lane == 0) sm.gpart[buf * SCAN_WARPS + warp] = gacc;
    __syncthreads();
    if (nbuf == 1) issue(i + 1);   // every thread is done with the single buffer
    // gate, refined scores (lane k: candidate k) and Select, identically in every warp
    float gate = a.b_g;
    for (int w = 0; w < SCAN_WARPS; ++w) gate += sm.gpart[buf * SCAN_WARPS + w];
#pragma unroll
    for (int f = 0; f < 5; ++f) gate = fmaf(wgf[f], phi[f], gate);
    const float gamma = sig_alpha * sigmoid_fast(gate);
    const float* clp = sm.clp + i * K;
    const float ref = lane < K ? clp[lane] + gamma * dot_k(red, lane) : -INFINITY;
    const int pick = select_warp(ref, K, a.select_mode, u_cur);
    if (warp == 0 && lane < K) {
      sm.ref[i * K + lane] = ref;
      a.refined[(bL + i) * K + lane] = ref;
    }
    if (a.select_mode == BRISK_SELECT_SAMPLE && i + 1 < L) u_cur = a.u_sel[bL + i + 1];
    prank = pick;
    prev = ci[pick];
    if (tid == 0) {
      sm.sel[i] = prev;
      sm.rank[i] = pick;
      a.sel_tokens[bL + i] = prev;
    }
  }
  if (timed_out && lane == 0) set_status(a.status, BRISK_ERR_TIMEOUT);
  // every copy that was issued has been waited for above (the last one at position L - 1)
}

__global__ void __launch_bounds__(SCAN_THREADS)
scan_kernel(const __grid_constant__ ScanArgs a) {
  extern __shared__ __align__(16) char smem_raw[];
  Smem sm;
  smem_layout(a.L, a.K, a.S, a.V, a.ubuf, a.tcand, smem_raw, &sm);
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  const int L = a.L, K = a.K, S = a.S, V = a.V;
  const size_t bL = (size_t)b * L;

  // Ids are gathered with below, so out-of-range ones (a row with no finite logit leaves
  // placeholder ids; caller-provided ids may be anything) are replaced by 0 and reported.
  for (int e = tid; e < L * K; e += SCAN_THREADS) {
    int c = a.cand_ids[bL * K + e];
    if (c < 0 || c >= V) { set_status(a.status, BRISK_ERR_NUMERIC); c = 0; }
    sm.cid[e] = c;
  }
  if (a.do_select) {
    for (int e = tid; e < L * K; e += SCAN_THREADS) sm.clp[e] = a.cand_logprob[bL * K + e];
  } else {
    for (int e = tid; e < L * K; e += SCAN_THREADS) sm.ref[e] = a.refined[bL * K + e];
    for (int e = tid; e < L; e += SCAN_THREADS) {
      int x = a.sel_tokens[bL + e];
      if (x < 0 || x >= V) { set_status(a.status, BRISK_ERR_INVALID_ARG); x = 0; }
      sm.sel[e] = x;
    }
  }
  __syncthreads();

  if (a.do_select) {
    int x0 = a.x0[b];
    if (x0 < 0 || x0 >= V) {
      if (tid == 0) set_status(a.status, BRISK_ERR_INVALID_ARG);
      x0 = 0;
    }
    // features' logit gathers, all independent of the selections
    for (int e = tid; e < L * 3; e += SCAN_THREADS) {
      const int i = e / 3, w = e % 3;
      const int c = sm.cid[i * K + (w == 0 ? 0 : (w == 1 ? 1 : 3))];
      sm.top[e] = load_logit(a.logits_q, a.logits_dt, (bL + i) * V + c);
    }
    for (int e = tid; e < L * K; e += SCAN_THREADS) {
      const int i = e / K, k = e % K;
      float v = 0.f;
      if (i == 0) { if (k == 0) v = load_logit(a.logits_q, a.logits_dt, bL * V + x0); }
      else v = load_logit(a.logits_q, a.logits_dt, (bL + i) * V + sm.cid[(i - 1) * K + k]);
      sm.lprev[e] = v;
    }
    for (int e = tid; e < 5 * S; e += SCAN_THREADS) {
      const int j = e / 5, f = e % 5;
      sm.F[f * S + j] = a.Fz[e];
      sm.F[(5 + f) * S + j] = a.Fh[e];
    }
    if (K + 1 <= 16) corrector_loop<16>(a, sm, b, x0);
    else corrector_loop<32>(a, sm, b, x0);
    __syncthreads();
  } else {
    // verify alone: recover each selection's rank in its candidate list
    for (int i = tid; i < L; i += SCAN_THREADS) {
      int r = 0;
      for (int k = 0; k < K; ++k)
        if (sm.cid[i * K + k] == sm.sel[i]) { r = k; break; }
      sm.rank[i] = r;
    }
    __syncthreads();
  }

  if (a.do_verify) verify_sequence(a, sm, b);
}

}  // namespace

constexpr size_t SCAN_SMEM_LIMIT = 227 * 1024;

// Shared-memory plan: stage the token-share rows and prefetch two positions ahead when that
// fits, else less.
void scan_plan(int L, int K, int S, int V, int* nbuf, int* tcand) {
  const int plans[5][2] = {{3, 1}, {2, 1}, {3, 0}, {2, 0}, {1, 0}};
  for (const auto& p : plans) {
    if (smem_layout(L, K, S, V, p[0], p[1], nullptr, nullptr) <= SCAN_SMEM_LIMIT) {
      *nbuf = p[0];
      *tcand = p[1];
      return;
    }
  }
  *nbuf = 1;
  *tcand = 0;
}

size_t scan_smem_bytes(int L, int K, int S, int V) {
  int ubuf, tcand;
  scan_plan(L, K, S, V, &ubuf, &tcand);
  return smem_layout(L, K, S, V, ubuf, tcand, nullptr, nullptr);
}

cudaError_t launch_scan(const ScanArgs& a_in, cudaStream_t stream) {
  ScanArgs a = a_in;
  scan_plan(a.L, a.K, a.S, a.V, &a.ubuf, &a.tcand);
  const size_t smem = smem_layout(a.L, a.K, a.S, a.V, a.ubuf, a.tcand, nullptr, nullptr);
  cudaError_t e = cudaFuncSetAttribute(scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  scan_kernel<<<a.B, SCAN_THREADS, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace brisk
