// C ABI of the decode tail: argument checks, workspace and table layouts, launches.
#include <cuda.h>

#include <deque>
#include <mutex>
#include <string.h>

#include "brisk_internal.cuh"

using namespace brisk;

namespace {

constexpr size_t ALIGN = 256;
inline size_t up(size_t x) { return (x + ALIGN - 1) / ALIGN * ALIGN; }

bool dims_ok(const brisk_dims* d) {
  if (!d) return false;
  if (d->B < 1 || d->L < 1 || d->L > 64) return false;
  if (d->K < 4 || d->K > 32 || d->V < d->K) return false;
  if (d->d < 8 || d->d % 8 != 0) return false;
  if (d->r < 16 || d->r > 512 || d->r % 16 != 0) return false;
  if ((d->logits_dtype != BRISK_DT_F32 && d->logits_dtype != BRISK_DT_BF16) ||
      (d->hidden_dtype != BRISK_DT_F32 && d->hidden_dtype != BRISK_DT_BF16))
    return false;
  if ((long long)d->B * d->L * d->V > (1LL << 40)) return false;
  return true;
}

inline size_t esize(int dt) { return dt == BRISK_DT_BF16 ? 2 : 4; }

// ---------------------------------------------------------------- workspace layout
enum TailSchedule { SCHEDULE_OVERLAP = 0, SCHEDULE_SEPARATE = 1, SCHEDULE_FUSED = 2 };
// Largest pair of logit tensors (bytes) for the fused small-batch schedule. Measured per block
// (direct calls / graph replays): one sequence (16 MB) 124.9 / 106.4 us separate, 117.7 / 102.5
// us fused; 16 sequences (259 MB, stochastic) 188.9 / 175.2 us separate, 243.6 / 210.6 fused.
constexpr size_t FUSE_MAX_BYTES = size_t(64) << 20;

struct WsLayout {
  size_t status, counters, part_val, part_id, part_m, part_s, argmax_p, lse_p;
  size_t cand_ids, cand_logprob, lse_q, sel, refined, Hm, G, G0, distill, base_rank, total;
  int nchunk_q, nchunk_p, KP;   // chunks per proposal row (row layout) and verifier row
  int mode_p;                   // layout of the verifier rows' sweep (SweepMode)
  int schedule;                 // TailSchedule of brisk_decode_tail
};

WsLayout ws_layout(const brisk_dims* d) {
  WsLayout w{};
  const size_t BL = (size_t)d->B * d->L;
  const size_t S = 2 * (size_t)d->r;
  w.nchunk_q = sweep_chunks((int)BL, d->V, d->logits_dtype, SWEEP_ROWS);
  // Schedule of the fused tail and the verifier rows' layout (every entry point sweeps the
  // verifier rows the same way, so that the fused and separate calls give the same bits):
  //  OVERLAP  one task per proposal row: verifier rows in the split layout, beside the corrector;
  //  FUSED    chunked proposal rows and both logit tensors within FUSE_MAX_BYTES: verifier rows
  //           in the row layout with the proposal rows' chunks, both tensors in one launch;
  //  SEPARATE chunked proposal rows, larger tensors: verifier rows in the split layout, beside
  //           the corrector (the verifier sweep then takes long enough that overlapping it with
  //           the corrector beats one launch before it).
  const size_t sweep_bytes = 2 * BL * (size_t)d->V * esize(d->logits_dtype);
  if (w.nchunk_q == 1) w.schedule = SCHEDULE_OVERLAP;
  else w.schedule = sweep_bytes <= FUSE_MAX_BYTES ? SCHEDULE_FUSED : SCHEDULE_SEPARATE;
  w.mode_p = w.schedule == SCHEDULE_FUSED ? SWEEP_ROWS : SWEEP_SPLIT;
  w.nchunk_p = w.schedule == SCHEDULE_FUSED
                   ? w.nchunk_q
                   : sweep_chunks((int)BL, d->V, d->logits_dtype, SWEEP_SPLIT);
  w.KP = kp_for(d->K);
  const size_t np = BL * (size_t)(w.nchunk_q + w.nchunk_p);
  size_t o = 0;
  auto take = [&](size_t bytes) { const size_t r = o; o = up(o + bytes); return r; };
  w.status = take(ALIGN);
  w.counters = take(sizeof(int32_t) * 2 * BL);
  w.part_val = take(sizeof(float) * np * w.KP);
  w.part_id = take(sizeof(int32_t) * np * w.KP);
  w.part_m = take(sizeof(float) * np);
  w.part_s = take(sizeof(float) * np);
  w.argmax_p = take(sizeof(int32_t) * BL);
  w.lse_p = take(sizeof(float) * BL);
  w.cand_ids = take(sizeof(int32_t) * BL * d->K);
  w.cand_logprob = take(sizeof(float) * BL * d->K);
  w.lse_q = take(sizeof(float) * BL);
  w.sel = take(sizeof(int32_t) * BL);
  w.refined = take(sizeof(float) * BL * d->K);
  w.Hm = take(6 * (BL + d->B) * d->r);   // fp32 [BL+B, r] or bf16 [BL+B, 3r]
  w.G = take(sizeof(float) * BL * 2 * S);
  w.G0 = take(sizeof(float) * d->B * S);
  w.distill = take(sizeof(float) * d->B);   // per-sequence loss partials of brisk_distill_loss
  w.base_rank = take(sizeof(int32_t) * BL);  // base selections of brisk_replay_diagnostics
  w.total = o;
  return w;
}

// ---------------------------------------------------------------- folded tables layout
// Tzh [V, 2S]: token share of the GRU pre-activations, Tz(v) | Th(v) with
//              Tz(v) = W_z[:, r:2r] P_e E_in(v), Th(v) = W_h[:, r:2r] P_e E_in(v)
// U   [V, S] : residual rows, U(v) = W_s^T W_c E_out(v)
// T0  [V, S] : token share of Init, W0[:, r:2r] P_e E_in(v)
// Tin, Tout [V, r]: P_e E_in(v), W_c E_out(v) (intermediates of the folds; on the tensor-core
//              path their space holds one of them at a time as three bf16 parts [V, 3r])
// posG [L, 2S]: position shares W_z[:, 2r:2r+16] pos_i | W_h[:, 2r:2r+16] pos_i
// Fz, Fh [S, 5]: feature shares W_z[:, 2r+16:] P_phi, W_h[:, 2r+16:] P_phi
// wg [S+5] fp32 copy of w_g; W2 [2S, r] = [W_z[:, :r] ; W_h[:, :r]] and W0h [S, r] = W0[:, :r] (fp32)
// W2s [2S, 3r], W0s [S, 3r] (bf16): the same blocks written three times along k, so that
// [hi | mid | lo] W^T = (hi + mid + lo) W^T on bf16 tensor cores.
struct TbLayout {
  size_t Tzh, U, T0, Tin, Tout, posG, Fz, Fh, wg, W2, W0h, W2s, W0s, Wt2s, W0ts, Ws3, total;
};

TbLayout tb_layout(const brisk_dims* d) {
  TbLayout t{};
  const size_t V = d->V, r = d->r, S = 2 * r, L = d->L;
  size_t o = 0;
  auto take = [&](size_t bytes) { const size_t q = o; o = up(o + bytes); return q; };
  t.Tzh = take(sizeof(float) * V * 2 * S);
  t.U = take(sizeof(float) * V * S);
  t.T0 = take(sizeof(float) * V * S);
  t.Tin = take(sizeof(float) * V * r);
  t.Tout = take(sizeof(float) * V * r);
  t.posG = take(sizeof(float) * L * 2 * S);
  t.Fz = take(sizeof(float) * S * 5);
  t.Fh = take(sizeof(float) * S * 5);
  t.wg = take(sizeof(float) * (S + 5));
  t.W2 = take(sizeof(float) * 2 * S * r);
  t.W0h = take(sizeof(float) * S * r);
  t.W2s = take(2 * 2 * S * 3 * r);
  t.W0s = take(2 * S * 3 * r);
  // bf16 token-side blocks written three times along k, for the folds on the tensor cores:
  // [W_z[:, r:2r] ; W_h[:, r:2r]] [2S, 3r], W0[:, r:2r] [S, 3r], W_s^T [S, 3r]
  t.Wt2s = take(2 * 2 * S * 3 * r);
  t.W0ts = take(2 * S * 3 * r);
  t.Ws3 = take(2 * S * 3 * r);
  t.total = o;
  return t;
}

template <typename T>
inline T* at(void* base, size_t off) { return reinterpret_cast<T*>(static_cast<char*>(base) + off); }
template <typename T>
inline const T* at(const void* base, size_t off) {
  return reinterpret_cast<const T*>(static_cast<const char*>(base) + off);
}

inline bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

#define BRISK_CUDA(call)                       \
  do {                                         \
    if ((call) != cudaSuccess) return BRISK_ERR_CUDA; \
  } while (0)

bool params_ok(const brisk_params* p) {
  return p && p->E_in && p->E_out && p->P_h && p->P_e && p->P_phi && p->pos && p->W0 && p->Wz &&
         p->Wh && p->W_s && p->W_c && p->w_g;
}

// Clears the status word and the sweep arrival counters of a workspace.
brisk_status clear_ws(const WsLayout& w, const brisk_dims* d, void* ws, cudaStream_t st) {
  BRISK_CUDA(cudaMemsetAsync(ws, 0, w.counters + sizeof(int32_t) * 2 * (size_t)d->B * d->L, st));
  return BRISK_OK;
}

SweepSeg make_seg(const WsLayout& w, void* ws, int seg, const void* logits, int rows, int kout,
                  int32_t* out_ids, float* out_logprob, float* out_lse) {
  SweepSeg s{};
  const size_t off = seg ? (size_t)rows * w.nchunk_q : 0;   // segment 1 follows segment 0
  s.logits = logits;
  s.rows = rows;
  s.kout = kout;
  s.out_ids = out_ids;
  s.out_logprob = out_logprob;
  s.out_lse = out_lse;
  s.part_val = at<float>(ws, w.part_val) + off * w.KP;
  s.part_id = at<int32_t>(ws, w.part_id) + off * w.KP;
  s.part_m = at<float>(ws, w.part_m) + off;
  s.part_s = at<float>(ws, w.part_s) + off;
  s.counters = at<int32_t>(ws, w.counters) + (size_t)seg * rows;
  return s;
}

// The hidden-state shares of the corrector: Hm = [hidden ; h_ctx] P_h^T, then
// G = Hm[:BL] [W_z[:, :r] ; W_h[:, :r]]^T and G0 = Hm[BL:] W0[:, :r]^T. With bf16 weights the
// products run on the tensor cores: the first one writes Hm as three bf16 parts, which the
// second one multiplies by the weight blocks written three times along k (fp32-level accuracy).
// The first product (k = d long) has few 128-row tiles for small batches: there it uses 64-wide
// column tiles and a 4-deep pipeline (four times the CTAs, each streaming a quarter of the
// weights). With `wide` (large batches, the products running beside the proposal sweep) it uses
// 256-wide tiles and a 2-deep pipeline: a quarter of the CTAs, so the sweep waits for fewer SMs,
// and the hidden states are read once; or, where the second product is small (S <= 512), both
// products in 64-wide tiles and a 2-deep pipeline that fit the sweep's shared-memory carveout,
// so that their CTAs share SMs with sweep CTAs instead of holding SMs of their own (decode_stream
// 395 -> 392 us a step; large_vocab's four times larger second product: 561 -> 601 us, not
// used there). Tile width does not change any product's summation order, so all give the same
// bits.
brisk_status hidden_products(const brisk_dims* d, const brisk_params* p, const void* tables,
                             const void* hidden, const void* h_ctx, const WsLayout& w, void* ws,
                             cudaStream_t st, bool wide) {
  const TbLayout t = tb_layout(d);
  const int BL = d->B * d->L, r = d->r, S = 2 * d->r, hd = d->hidden_dtype;
  int32_t* status = at<int32_t>(ws, w.status);
  if (hd == BRISK_DT_BF16 && gemm_tc_supported(hidden, d->d, p->P_h, d->d, d->d) &&
      aligned(h_ctx, 16)) {
    __nv_bfloat16* Hs = at<__nv_bfloat16>(ws, w.Hm);   // [BL + B, 3r]: hi | mid | lo
    const int r3 = 3 * r;
    const bool share = wide && S <= 512;   // tiles that fit the sweep's carveout
    const int bn = wide && !share ? 256 : 64;
    const TcSpec first[2] = {
        {BL, r, d->d, hidden, d->d, p->P_h, d->d, 1, Hs, r3, nullptr, 0, bn},
        {d->B, r, d->d, h_ctx, d->d, p->P_h, d->d, 1, Hs + (size_t)BL * r3, r3, nullptr, 0, bn}};
    BRISK_CUDA(gemm_tc_grouped(first, 2, status, st, wide ? 2 : 4, share));
    const TcSpec second[2] = {
        {BL, 2 * S, r3, Hs, r3, at<__nv_bfloat16>(tables, t.W2s), r3, 0, at<float>(ws, w.G), 2 * S,
         nullptr, 0, share ? 64 : 0},
        {d->B, S, r3, Hs + (size_t)BL * r3, r3, at<__nv_bfloat16>(tables, t.W0s), r3, 0,
         at<float>(ws, w.G0), S, nullptr, 0, share ? 64 : 0}};
    BRISK_CUDA(gemm_tc_grouped(second, 2, status, st, 2, share));
    return BRISK_OK;
  }
  float* Hm = at<float>(ws, w.Hm);
  BRISK_CUDA(gemm_simt(BL, r, d->d, hidden, hd, d->d, p->P_h, hd, d->d, false, Hm, r, st));
  BRISK_CUDA(gemm_simt(d->B, r, d->d, h_ctx, hd, d->d, p->P_h, hd, d->d, false,
                       Hm + (size_t)BL * r, r, st));
  BRISK_CUDA(gemm_simt(BL, 2 * S, r, Hm, BRISK_DT_F32, r, at<float>(tables, t.W2), BRISK_DT_F32, r,
                       false, at<float>(ws, w.G), 2 * S, st));
  BRISK_CUDA(gemm_simt(d->B, S, r, Hm + (size_t)BL * r, BRISK_DT_F32, r, at<float>(tables, t.W0h),
                       BRISK_DT_F32, r, false, at<float>(ws, w.G0), S, st));
  return BRISK_OK;
}

// Side streams per CUDA context (created on the first fused call in that context, so a device
// reset gets new ones) and the events that fork work onto them and join it back, so that one
// call can run independent stages concurrently.
struct SideStream {
  unsigned long long ctx = 0;   // id of the context the streams belong to
  cudaStream_t hi = nullptr;    // highest priority: the hidden-state products
  cudaStream_t mid = nullptr;   // middle priority: proposal sweep, corrector, verification
  cudaStream_t lo = nullptr;    // lowest priority: the verifier-row sweep
  cudaEvent_t ev[5] = {};
};
std::deque<SideStream> g_side;   // guarded by side_stream_mutex(); elements never move

// The current context's side streams; the caller holds side_stream_mutex().
SideStream* side_stream() {
  unsigned long long ctx = 0;
  if (!brisk::current_context_id(&ctx)) return nullptr;
  SideStream* found = nullptr;
  for (auto& e : g_side)
    if (e.ctx == ctx) found = &e;
  if (!found) {
    g_side.emplace_back();
    found = &g_side.back();
    found->ctx = ctx;
  }
  SideStream& ss = *found;
  if (!ss.hi) {
    int least = 0, greatest = 0;
    if (cudaDeviceGetStreamPriorityRange(&least, &greatest) != cudaSuccess) return nullptr;
    cudaStream_t hi = nullptr, mid = nullptr, lo = nullptr;
    if (cudaStreamCreateWithPriority(&hi, cudaStreamNonBlocking, greatest) != cudaSuccess ||
        cudaStreamCreateWithPriority(&mid, cudaStreamNonBlocking, (least + greatest) / 2) !=
            cudaSuccess ||
        cudaStreamCreateWithPriority(&lo, cudaStreamNonBlocking, least) != cudaSuccess)
      return nullptr;
    for (auto& e : ss.ev)
      if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return nullptr;
    ss.lo = lo;
    ss.mid = mid;
    ss.hi = hi;
  }
  return &ss;
}

ScanArgs scan_args(const brisk_dims* d, const brisk_params* p, const void* tables, const WsLayout& w,
                   void* ws) {
  ScanArgs a{};
  a.B = d->B; a.L = d->L; a.V = d->V; a.K = d->K; a.S = 2 * d->r; a.logits_dt = d->logits_dtype;
  a.status = at<int32_t>(ws, w.status);
  if (tables) {
    const TbLayout t = tb_layout(d);
    a.Tzh = at<float>(tables, t.Tzh);
    a.posG = at<float>(tables, t.posG);
    a.U = at<float>(tables, t.U);
    a.T0 = at<float>(tables, t.T0);
    a.Fz = at<float>(tables, t.Fz);
    a.Fh = at<float>(tables, t.Fh);
    a.wg = at<float>(tables, t.wg);
  }
  if (p) {
    a.b_g = p->b_g;
    a.alpha = p->alpha;
  }
  a.G = at<float>(ws, w.G);
  a.G0 = at<float>(ws, w.G0);
  a.argmax_p = at<int32_t>(ws, w.argmax_p);
  a.lse_p = at<float>(ws, w.lse_p);
  return a;
}

}  // namespace

std::mutex& brisk::side_stream_mutex() {
  static std::mutex mu;
  return mu;
}

bool brisk::current_context_id(unsigned long long* id) {
  using GetCurrent = CUresult (*)(CUcontext*);
  using GetId = CUresult (*)(CUcontext, unsigned long long*);
  static GetCurrent get_current = nullptr;
  static GetId get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrent>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetId>(p);
  });
  if (!get_current || !get_id) return false;
  CUcontext c = nullptr;
  if (get_current(&c) != CUDA_SUCCESS || !c) return false;
  return get_id(c, id) == CUDA_SUCCESS;
}

extern "C" {

size_t brisk_workspace_bytes(const brisk_dims* dims) {
  if (!dims_ok(dims)) return 0;
  return ws_layout(dims).total;
}

size_t brisk_tables_bytes(const brisk_dims* dims) {
  if (!dims_ok(dims)) return 0;
  return tb_layout(dims).total;
}

const char* brisk_status_string(brisk_status s) {
  switch (s) {
    case BRISK_OK: return "BRISK_OK";
    case BRISK_ERR_INVALID_ARG: return "BRISK_ERR_INVALID_ARG";
    case BRISK_ERR_UNSUPPORTED: return "BRISK_ERR_UNSUPPORTED";
    case BRISK_ERR_CUDA: return "BRISK_ERR_CUDA";
    case BRISK_ERR_TIMEOUT: return "BRISK_ERR_TIMEOUT";
    case BRISK_ERR_NUMERIC: return "BRISK_ERR_NUMERIC";
  }
  return "BRISK_ERR_UNKNOWN";
}

brisk_status brisk_corrector_prepare(const brisk_dims* d, const brisk_params* p, void* tables,
                                     void* stream) {
  if (!dims_ok(d) || !params_ok(p) || !tables || !aligned(tables, ALIGN)) return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const TbLayout t = tb_layout(d);
  const int V = d->V, r = d->r, S = 2 * r, L = d->L, hd = d->hidden_dtype, F32 = BRISK_DT_F32;
  const int ldw = 2 * r + 32;
  const size_t es = esize(hd);
  auto wp = [&](const void* base, size_t elems) {
    return static_cast<const void*>(static_cast<const char*>(base) + elems * es);
  };
  float* Tin = at<float>(tables, t.Tin);
  float* Tout = at<float>(tables, t.Tout);
  float* Tzh = at<float>(tables, t.Tzh);
  if (hd == BRISK_DT_BF16 && gemm_tc_supported(p->E_in, d->d, p->P_e, d->d, d->d) &&
      gemm_tc_supported(p->E_out, d->d, p->W_c, d->d, d->d)) {
    // On the tensor cores. P_e E_in(v) (then W_c E_out(v)) is written as three bf16 parts
    // (hi + mid + lo, exact to about 2^-24 relative) into the Tin / Tout space, and the next
    // products multiply the parts by the weight blocks written three times along k, which keeps
    // fp32-level accuracy on bf16 tensor cores. No status word: a bounded wait that gives up
    // here (about 2 s at the default limit) leaves the tables undefined.
    const int BF = BRISK_DT_BF16, r3 = 3 * r;
    __nv_bfloat16* Wt2s = at<__nv_bfloat16>(tables, t.Wt2s);
    __nv_bfloat16* W0ts = at<__nv_bfloat16>(tables, t.W0ts);
    __nv_bfloat16* Ws3 = at<__nv_bfloat16>(tables, t.Ws3);
    for (int part = 0; part < 3; ++part) {
      BRISK_CUDA(copy2d(S, r, wp(p->Wz, r), hd, ldw, Wt2s + part * r, BF, r3, st));
      BRISK_CUDA(copy2d(S, r, wp(p->Wh, r), hd, ldw, Wt2s + (size_t)S * r3 + part * r, BF, r3, st));
      BRISK_CUDA(copy2d(S, r, wp(p->W0, r), hd, 2 * r, W0ts + part * r, BF, r3, st));
      BRISK_CUDA(copy2d(S, r, p->W_s, hd, S, Ws3 + part * r, BF, r3, st, true));   // W_s^T
    }
    __nv_bfloat16* X3 = at<__nv_bfloat16>(tables, t.Tin);   // [V, 3r] in the Tin and Tout space
    BRISK_CUDA(gemm_tc(V, r, d->d, p->E_in, d->d, p->P_e, d->d, 1, X3, r3, nullptr, st));
    const TcSpec tok[2] = {{V, 2 * S, r3, X3, r3, Wt2s, r3, 0, Tzh, 2 * S, nullptr, 0, 0},
                           {V, S, r3, X3, r3, W0ts, r3, 0, at<float>(tables, t.T0), S, nullptr, 0, 0}};
    BRISK_CUDA(gemm_tc_grouped(tok, 2, nullptr, st, 4));
    BRISK_CUDA(gemm_tc(V, r, d->d, p->E_out, d->d, p->W_c, d->d, 1, X3, r3, nullptr, st));
    BRISK_CUDA(gemm_tc(V, S, r3, X3, r3, Ws3, r3, 0, at<float>(tables, t.U), S, nullptr, st));
  } else {
    // P_e E_in(v) and W_c E_out(v) for every v
    BRISK_CUDA(gemm_simt(V, r, d->d, p->E_in, hd, d->d, p->P_e, hd, d->d, false, Tin, r, st));
    BRISK_CUDA(gemm_simt(V, r, d->d, p->E_out, hd, d->d, p->W_c, hd, d->d, false, Tout, r, st));
    // token shares of the gate / candidate pre-activations and of Init
    BRISK_CUDA(gemm_simt(V, S, r, Tin, F32, r, wp(p->Wz, r), hd, ldw, false, Tzh, 2 * S, st));
    BRISK_CUDA(gemm_simt(V, S, r, Tin, F32, r, wp(p->Wh, r), hd, ldw, false, Tzh + S, 2 * S, st));
    BRISK_CUDA(gemm_simt(V, S, r, Tin, F32, r, wp(p->W0, r), hd, 2 * r, false,
                         at<float>(tables, t.T0), S, st));
    // residual rows U(v) = W_s^T (W_c E_out(v)): B(n=j, k=t) = W_s[t, j]
    BRISK_CUDA(gemm_simt(V, S, r, Tout, F32, r, p->W_s, hd, S, true, at<float>(tables, t.U), S, st));
  }
  // position shares
  BRISK_CUDA(gemm_simt(L, S, 16, p->pos, hd, 16, wp(p->Wz, 2 * r), hd, ldw, false,
                       at<float>(tables, t.posG), 2 * S, st));
  BRISK_CUDA(gemm_simt(L, S, 16, p->pos, hd, 16, wp(p->Wh, 2 * r), hd, ldw, false,
                       at<float>(tables, t.posG) + S, 2 * S, st));
  // feature shares: F(j, f) = sum_t W[j, 2r+16+t] P_phi[t, f]
  BRISK_CUDA(gemm_simt(S, 5, 16, wp(p->Wz, 2 * r + 16), hd, ldw, p->P_phi, hd, 5, true,
                       at<float>(tables, t.Fz), 5, st));
  BRISK_CUDA(gemm_simt(S, 5, 16, wp(p->Wh, 2 * r + 16), hd, ldw, p->P_phi, hd, 5, true,
                       at<float>(tables, t.Fh), 5, st));
  // fp32 copies of the gate weights and of the hidden-state blocks
  BRISK_CUDA(copy2d(1, S + 5, p->w_g, hd, S + 5, at<float>(tables, t.wg), F32, S + 5, st));
  BRISK_CUDA(copy2d(S, r, p->Wz, hd, ldw, at<float>(tables, t.W2), F32, r, st));
  BRISK_CUDA(copy2d(S, r, p->Wh, hd, ldw, at<float>(tables, t.W2) + (size_t)S * r, F32, r, st));
  BRISK_CUDA(copy2d(S, r, p->W0, hd, 2 * r, at<float>(tables, t.W0h), F32, r, st));
  if (hd == BRISK_DT_BF16) {
    const int BF = BRISK_DT_BF16;
    __nv_bfloat16* W2s = at<__nv_bfloat16>(tables, t.W2s);
    __nv_bfloat16* W0s = at<__nv_bfloat16>(tables, t.W0s);
    for (int part = 0; part < 3; ++part) {
      BRISK_CUDA(copy2d(S, r, p->Wz, hd, ldw, W2s + part * r, BF, 3 * r, st));
      BRISK_CUDA(copy2d(S, r, p->Wh, hd, ldw, W2s + (size_t)S * 3 * r + part * r, BF, 3 * r, st));
      BRISK_CUDA(copy2d(S, r, p->W0, hd, 2 * r, W0s + part * r, BF, 3 * r, st));
    }
  }
  return BRISK_OK;
}

brisk_status brisk_topk_candidates(const brisk_dims* d, const void* logits_q, int32_t* cand_ids,
                                   float* cand_logprob, float* lse_q, void* ws, void* stream) {
  if (!dims_ok(d) || !logits_q || !cand_ids || !cand_logprob || !lse_q || !ws ||
      !aligned(ws, ALIGN) || !aligned(logits_q, esize(d->logits_dtype)))
    return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const WsLayout w = ws_layout(d);
  brisk_status s = clear_ws(w, d, ws, st);
  if (s != BRISK_OK) return s;
  SweepLaunch a{};
  a.seg[0] = make_seg(w, ws, 0, logits_q, d->B * d->L, d->K, cand_ids, cand_logprob, lse_q);
  a.nseg = 1;
  a.V = d->V;
  a.mode = SWEEP_ROWS;
  a.nchunk = w.nchunk_q;
  a.KP = w.KP;
  a.dtype = d->logits_dtype;
  a.status = at<int32_t>(ws, w.status);
  BRISK_CUDA(launch_sweep(a, st));
  return BRISK_OK;
}

brisk_status brisk_corrector_select(const brisk_dims* d, const brisk_params* p, const void* tables,
                                    const void* hidden, const void* h_ctx, const int32_t* x0,
                                    const void* logits_q, const int32_t* cand_ids,
                                    const float* cand_logprob, int32_t select_mode,
                                    const float* u_sel, int32_t* sel_tokens, float* refined,
                                    void* ws, void* stream) {
  if (!dims_ok(d) || !params_ok(p) || !tables || !hidden || !h_ctx || !x0 || !logits_q ||
      !cand_ids || !cand_logprob || !sel_tokens || !refined || !ws || !aligned(ws, ALIGN) ||
      !aligned(tables, ALIGN))
    return BRISK_ERR_INVALID_ARG;
  if (select_mode != BRISK_SELECT_GREEDY && select_mode != BRISK_SELECT_SAMPLE)
    return BRISK_ERR_INVALID_ARG;
  if (select_mode == BRISK_SELECT_SAMPLE && !u_sel) return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const WsLayout w = ws_layout(d);
  brisk_status s = clear_ws(w, d, ws, st);
  if (s != BRISK_OK) return s;
  s = hidden_products(d, p, tables, hidden, h_ctx, w, ws, st, false);
  if (s != BRISK_OK) return s;
  ScanArgs a = scan_args(d, p, tables, w, ws);
  a.select_mode = select_mode;
  a.do_select = 1;
  a.do_verify = 0;
  a.logits_q = logits_q;
  a.cand_ids = cand_ids;
  a.cand_logprob = cand_logprob;
  a.x0 = x0;
  a.u_sel = u_sel;
  a.sel_tokens = sel_tokens;
  a.refined = refined;
  BRISK_CUDA(launch_scan(a, st));
  return BRISK_OK;
}

brisk_status brisk_verify_block(const brisk_dims* d, const void* logits_p, const int32_t* sel_tokens,
                                const int32_t* cand_ids, const float* refined, int32_t select_mode,
                                int32_t verify_mode, const float* u_acc, const float* u_res,
                                int32_t* accepted_len, int32_t* out_tokens, int32_t* correction,
                                void* ws, void* stream) {
  if (!dims_ok(d) || !logits_p || !sel_tokens || !cand_ids || !refined || !accepted_len ||
      !out_tokens || !correction || !ws || !aligned(ws, ALIGN) ||
      !aligned(logits_p, esize(d->logits_dtype)))
    return BRISK_ERR_INVALID_ARG;
  if ((select_mode != BRISK_SELECT_GREEDY && select_mode != BRISK_SELECT_SAMPLE) ||
      (verify_mode != BRISK_VERIFY_GREEDY && verify_mode != BRISK_VERIFY_STOCHASTIC))
    return BRISK_ERR_INVALID_ARG;
  if (verify_mode == BRISK_VERIFY_STOCHASTIC && (!u_acc || !u_res)) return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const WsLayout w = ws_layout(d);
  brisk_status s = clear_ws(w, d, ws, st);
  if (s != BRISK_OK) return s;
  SweepLaunch sw{};
  const int BL = d->B * d->L;
  sw.seg[0] = make_seg(w, ws, 1, logits_p, BL, 1, at<int32_t>(ws, w.argmax_p), nullptr,
                       at<float>(ws, w.lse_p));
  sw.nseg = 1;
  sw.V = d->V;
  sw.mode = w.mode_p;
  sw.nchunk = w.nchunk_p;
  sw.KP = w.KP;
  sw.dtype = d->logits_dtype;
  sw.status = at<int32_t>(ws, w.status);
  BRISK_CUDA(launch_sweep(sw, st));
  ScanArgs a = scan_args(d, nullptr, nullptr, w, ws);
  a.select_mode = select_mode;
  a.verify_mode = verify_mode;
  a.do_select = 0;
  a.do_verify = 1;
  a.cand_ids = cand_ids;
  a.sel_tokens = const_cast<int32_t*>(sel_tokens);
  a.refined = const_cast<float*>(refined);
  a.logits_p = logits_p;
  a.u_acc = u_acc;
  a.u_res = u_res;
  a.accepted_len = accepted_len;
  a.out_tokens = out_tokens;
  a.correction = correction;
  BRISK_CUDA(launch_scan(a, st));
  return BRISK_OK;
}

brisk_status brisk_decode_tail(const brisk_dims* d, const brisk_params* p, const void* tables,
                               const brisk_tail_io* io, int32_t select_mode, int32_t verify_mode,
                               void* ws, const brisk_events* ev, void* stream) {
  std::lock_guard<std::mutex> lock(side_stream_mutex());
  return brisk::decode_tail_locked(d, p, tables, io, select_mode, verify_mode, ws, ev, stream);
}

}  // extern "C"

// The body of brisk_decode_tail; the caller holds side_stream_mutex() (brisk_tail_graph_create
// holds it from the start of its capture to the end, so that no other thread's work lands on
// the side streams while they belong to the capture).
brisk_status brisk::decode_tail_locked(const brisk_dims* d, const brisk_params* p,
                                       const void* tables, const brisk_tail_io* io,
                                       int32_t select_mode, int32_t verify_mode, void* ws,
                                       const brisk_events* ev, void* stream) {
  if (!dims_ok(d) || !params_ok(p) || !tables || !io || !ws || !aligned(ws, ALIGN) ||
      !aligned(tables, ALIGN))
    return BRISK_ERR_INVALID_ARG;
  if (!io->logits_q || !io->logits_p || !io->hidden || !io->h_ctx || !io->x0 || !io->accepted_len ||
      !io->out_tokens || !io->correction)
    return BRISK_ERR_INVALID_ARG;
  if (!aligned(io->logits_q, esize(d->logits_dtype)) || !aligned(io->logits_p, esize(d->logits_dtype)))
    return BRISK_ERR_INVALID_ARG;
  if ((select_mode != BRISK_SELECT_GREEDY && select_mode != BRISK_SELECT_SAMPLE) ||
      (verify_mode != BRISK_VERIFY_GREEDY && verify_mode != BRISK_VERIFY_STOCHASTIC))
    return BRISK_ERR_INVALID_ARG;
  if (select_mode == BRISK_SELECT_SAMPLE && !io->u_sel) return BRISK_ERR_INVALID_ARG;
  if (verify_mode == BRISK_VERIFY_STOCHASTIC && (!io->u_acc || !io->u_res)) return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const WsLayout w = ws_layout(d);
  brisk_status s = clear_ws(w, d, ws, st);
  if (s != BRISK_OK) return s;
  const int BL = d->B * d->L;
  int32_t* cand_ids = io->cand_ids ? io->cand_ids : at<int32_t>(ws, w.cand_ids);
  float* cand_lp = io->cand_logprob ? io->cand_logprob : at<float>(ws, w.cand_logprob);
  float* lse_q = io->lse_q ? io->lse_q : at<float>(ws, w.lse_q);
  int32_t* sel = io->sel_tokens ? io->sel_tokens : at<int32_t>(ws, w.sel);
  float* refined = io->refined ? io->refined : at<float>(ws, w.refined);

  // Schedule on side streams forked from the caller's stream A, by priority:
  //   H (highest): hidden products -----.
  //   M (middle) : proposal sweep ---- join -> corrector --- join -> verification -> join A
  //   W (lowest) : verifier sweep ---------------------------'
  // The block scheduler places ready blocks of higher priority first. The products take their
  // SMs first; the proposal sweep, on the critical path (proposal candidates -> corrector ->
  // verification), takes the rest; the verifier sweep, needed only by the verification, starts
  // at once but only fills room the other two leave: the proposal sweep's ragged end (one
  // long task per row, ending over tens of microseconds) and the SMs beside the corrector.
  // In this mode the products use wide tiles (fewer SMs held at the start).
  // With chunked proposal rows (few rows) the short tasks end together and the critical path
  // stays on A, the products (on the critical path there) using narrow tiles (more CTAs):
  //  SEPARATE the verifier sweep starts after the proposal sweep, beside the corrector, which
  //           saves the extra fork and keeps the SMs free for the corrector's start;
  //  FUSED    (small tensors) one sweep launch on A covers the rows of both tensors, and the
  //           corrector that follows it verifies its sequence in the same CTA (four launches
  //           with two products, against six).
  const bool overlap = w.schedule == SCHEDULE_OVERLAP;
  SideStream* ss = side_stream();
  if (!ss) return BRISK_ERR_CUDA;
  cudaStream_t m = overlap ? ss->mid : st;
  BRISK_CUDA(cudaEventRecord(ss->ev[0], st));
  BRISK_CUDA(cudaStreamWaitEvent(ss->hi, ss->ev[0], 0));
  if (overlap) BRISK_CUDA(cudaStreamWaitEvent(m, ss->ev[0], 0));
  if (w.schedule != SCHEDULE_FUSED) BRISK_CUDA(cudaStreamWaitEvent(ss->lo, ss->ev[0], 0));
  s = hidden_products(d, p, tables, io->hidden, io->h_ctx, w, ws, ss->hi, overlap);
  if (s != BRISK_OK) return s;
  BRISK_CUDA(cudaEventRecord(ss->ev[1], ss->hi));

  SweepLaunch sq{};
  sq.seg[0] = make_seg(w, ws, 0, io->logits_q, BL, d->K, cand_ids, cand_lp, lse_q);
  sq.nseg = 1;
  sq.V = d->V;
  sq.mode = SWEEP_ROWS;
  sq.nchunk = w.nchunk_q;
  sq.KP = w.KP;
  sq.dtype = d->logits_dtype;
  sq.status = at<int32_t>(ws, w.status);
  SweepLaunch sp = sq;
  sp.seg[0] = make_seg(w, ws, 1, io->logits_p, BL, 1, at<int32_t>(ws, w.argmax_p), nullptr,
                       at<float>(ws, w.lse_p));
  sp.mode = w.mode_p;
  sp.nchunk = w.nchunk_p;
  ScanArgs a = scan_args(d, p, tables, w, ws);
  a.select_mode = select_mode;
  a.verify_mode = verify_mode;
  a.do_select = 1;
  a.do_verify = 0;
  a.logits_q = io->logits_q;
  a.cand_ids = cand_ids;
  a.cand_logprob = cand_lp;
  a.x0 = io->x0;
  a.u_sel = io->u_sel;
  a.sel_tokens = sel;
  a.refined = refined;

  if (w.schedule == SCHEDULE_FUSED) {
    // both tensors' rows in one launch (the same layout and chunks as the separate calls)
    SweepLaunch both = sq;
    both.seg[1] = sp.seg[0];
    both.nseg = 2;
    if (ev && ev->sweep_q_begin) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_q_begin), st));
    if (ev && ev->sweep_p_begin) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_p_begin), st));
    BRISK_CUDA(launch_sweep(both, st));
    if (ev && ev->sweep_q_end) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_q_end), st));
    if (ev && ev->sweep_p_end) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_p_end), st));
    // the corrector once the hidden products are done, verifying in the same CTA
    BRISK_CUDA(cudaStreamWaitEvent(st, ss->ev[1], 0));
    a.do_verify = 1;
    a.logits_p = io->logits_p;
    a.u_acc = io->u_acc;
    a.u_res = io->u_res;
    a.accepted_len = io->accepted_len;
    a.out_tokens = io->out_tokens;
    a.correction = io->correction;
    a.next_anchor = io->next_anchor;
    BRISK_CUDA(launch_scan(a, st));
    return BRISK_OK;
  }

  if (ev && ev->sweep_q_begin) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_q_begin), m));
  BRISK_CUDA(launch_sweep(sq, m));
  if (ev && ev->sweep_q_end) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_q_end), m));
  if (!overlap) {
    // SEPARATE: the verifier rows after the proposal rows, beside the corrector
    BRISK_CUDA(cudaEventRecord(ss->ev[2], m));
    BRISK_CUDA(cudaStreamWaitEvent(ss->lo, ss->ev[2], 0));
  }

  // verifier rows on the low-priority stream
  if (ev && ev->sweep_p_begin) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_p_begin), ss->lo));
  BRISK_CUDA(launch_sweep(sp, ss->lo));
  // the join first: a timing record ahead of it would delay the verification behind it
  BRISK_CUDA(cudaEventRecord(ss->ev[3], ss->lo));
  if (ev && ev->sweep_p_end) BRISK_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ev->sweep_p_end), ss->lo));

  // the corrector once the proposal candidates and the hidden products are done
  BRISK_CUDA(cudaStreamWaitEvent(m, ss->ev[1], 0));
  BRISK_CUDA(launch_scan(a, m));
  BRISK_CUDA(cudaStreamWaitEvent(m, ss->ev[3], 0));

  ScanArgs v = scan_args(d, nullptr, nullptr, w, ws);
  v.select_mode = select_mode;
  v.verify_mode = verify_mode;
  v.do_select = 0;
  v.do_verify = 1;
  v.cand_ids = cand_ids;
  v.sel_tokens = sel;
  v.refined = refined;
  v.logits_p = io->logits_p;
  v.u_acc = io->u_acc;
  v.u_res = io->u_res;
  v.accepted_len = io->accepted_len;
  v.out_tokens = io->out_tokens;
  v.correction = io->correction;
  v.next_anchor = io->next_anchor;
  BRISK_CUDA(launch_scan(v, m));
  if (overlap) {
    BRISK_CUDA(cudaEventRecord(ss->ev[4], m));
    BRISK_CUDA(cudaStreamWaitEvent(st, ss->ev[4], 0));
  }
  return BRISK_OK;
}

extern "C" {

int32_t brisk_kernels_per_tail(const brisk_dims* dims) {
  if (!dims_ok(dims)) return 0;
  const bool tc = dims->hidden_dtype == BRISK_DT_BF16;
  const int products = tc ? 2 : 4;
  // two sweeps, the products, the corrector, the verification; in the fused small-batch
  // schedule one sweep of both tensors, the products, the corrector that also verifies
  if (ws_layout(dims).schedule != SCHEDULE_FUSED) return 2 + products + 1 + 1;
  return 1 + products + 1;
}

brisk_status brisk_last_device_status(void* ws, int32_t clear, void* stream) {
  if (!ws) return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t h = 0;
  BRISK_CUDA(cudaMemcpyAsync(&h, ws, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  BRISK_CUDA(cudaStreamSynchronize(st));
  if (clear) {
    BRISK_CUDA(cudaMemsetAsync(ws, 0, sizeof(int32_t), st));
    BRISK_CUDA(cudaStreamSynchronize(st));
  }
  return static_cast<brisk_status>(h);
}


brisk_status brisk_distill_loss(const brisk_dims* d, const void* logits_p, const int32_t* cand_ids,
                                const float* cand_logprob, const float* refined,
                                const int32_t* accepted_len, float beta, float* loss,
                                float* grad_refined, void* ws, void* stream) {
  if (!dims_ok(d) || !logits_p || !cand_ids || !cand_logprob || !refined || !accepted_len ||
      !loss || !ws || !aligned(ws, ALIGN) || !aligned(logits_p, esize(d->logits_dtype)) ||
      !(beta >= 0.f))
    return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const WsLayout w = ws_layout(d);
  brisk_status s = clear_ws(w, d, ws, st);
  if (s != BRISK_OK) return s;
  DistillArgs a{};
  a.B = d->B; a.L = d->L; a.V = d->V; a.K = d->K; a.logits_dt = d->logits_dtype;
  a.logits_p = logits_p;
  a.cand_ids = cand_ids;
  a.cand_logprob = cand_logprob;
  a.refined = refined;
  a.accepted_len = accepted_len;
  a.beta = beta;
  a.loss = loss;
  a.grad = grad_refined;
  a.partial = at<float>(ws, w.distill);
  a.arrivals = at<int32_t>(ws, w.status) + 16;   // a word of the (cleared) status block
  a.status = at<int32_t>(ws, w.status);
  BRISK_CUDA(launch_distill(a, st));
  return BRISK_OK;
}

brisk_status brisk_replay_diagnostics(const brisk_dims* d, const brisk_params* p, const void* tables,
                                      const void* hidden, const void* h_ctx, const int32_t* x0,
                                      const void* logits_q, const void* logits_p,
                                      int32_t select_mode, const float* u_sel, const float* u_acc,
                                      int32_t* head_tokens, int32_t* flags,
                                      int32_t* first_breaker, float* refined, void* ws,
                                      void* stream) {
  if (!dims_ok(d) || !params_ok(p) || !tables || !hidden || !h_ctx || !x0 || !logits_q ||
      !logits_p || !u_acc || !head_tokens || !flags || !first_breaker || !ws ||
      !aligned(ws, ALIGN) || !aligned(tables, ALIGN) || !aligned(logits_q, esize(d->logits_dtype)) ||
      !aligned(logits_p, esize(d->logits_dtype)))
    return BRISK_ERR_INVALID_ARG;
  if (select_mode != BRISK_SELECT_GREEDY && select_mode != BRISK_SELECT_SAMPLE)
    return BRISK_ERR_INVALID_ARG;
  if (select_mode == BRISK_SELECT_SAMPLE && !u_sel) return BRISK_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const WsLayout w = ws_layout(d);
  brisk_status s = clear_ws(w, d, ws, st);
  if (s != BRISK_OK) return s;
  const int BL = d->B * d->L;
  int32_t* cand_ids = at<int32_t>(ws, w.cand_ids);
  float* cand_lp = at<float>(ws, w.cand_logprob);
  float* ref = refined ? refined : at<float>(ws, w.refined);
  // candidates, and the verifier rows' log-partition
  SweepLaunch sq{};
  sq.seg[0] = make_seg(w, ws, 0, logits_q, BL, d->K, cand_ids, cand_lp, at<float>(ws, w.lse_q));
  sq.nseg = 1;
  sq.V = d->V;
  sq.mode = SWEEP_ROWS;
  sq.nchunk = w.nchunk_q;
  sq.KP = w.KP;
  sq.dtype = d->logits_dtype;
  sq.status = at<int32_t>(ws, w.status);
  BRISK_CUDA(launch_sweep(sq, st));
  SweepLaunch sp = sq;
  sp.seg[0] = make_seg(w, ws, 1, logits_p, BL, 1, at<int32_t>(ws, w.argmax_p), nullptr,
                       at<float>(ws, w.lse_p));
  sp.mode = w.mode_p;
  sp.nchunk = w.nchunk_p;
  BRISK_CUDA(launch_sweep(sp, st));
  // the head along the factual base prefix
  s = hidden_products(d, p, tables, hidden, h_ctx, w, ws, st, false);
  if (s != BRISK_OK) return s;
  ScanArgs a = scan_args(d, p, tables, w, ws);
  a.select_mode = select_mode;
  a.do_select = 1;
  a.logits_q = logits_q;
  a.cand_ids = cand_ids;
  a.cand_logprob = cand_lp;
  a.x0 = x0;
  a.u_sel = u_sel;
  a.sel_tokens = head_tokens;
  a.refined = ref;
  a.base_prefix = 1;
  a.base_rank = at<int32_t>(ws, w.base_rank);
  BRISK_CUDA(launch_scan(a, st));
  ReplayArgs r{};
  r.B = d->B; r.L = d->L; r.V = d->V; r.K = d->K; r.logits_dt = d->logits_dtype;
  r.logits_p = logits_p;
  r.lse_p = at<float>(ws, w.lse_p);
  r.cand_ids = cand_ids;
  r.cand_logprob = cand_lp;
  r.base_rank = a.base_rank;
  r.head_tokens = head_tokens;
  r.u_acc = u_acc;
  r.flags = flags;
  r.first_breaker = first_breaker;
  r.status = at<int32_t>(ws, w.status);
  BRISK_CUDA(launch_replay(r, st));
  return BRISK_OK;
}

}  // extern "C"
