/*
 * brisk.h - C ABI of the BRISK-DLM per-block decode tail on GB300 (sm_103a).
 *
 * The decode tail turns one backbone evaluation of a diffusion language model
 * into verified tokens (paper: "From Position Risks to Block Survival: Faster
 * Generation for Diffusion Language Models", Sec. 3.3 and Algorithm 1(b)):
 *
 *   1. candidates: log-sum-exp over the full vocabulary and the ordered Top-K
 *      of every masked position (Sec. 3.3 "C_i = TopK(q_i, K)"; App. C.3);
 *   2. the prefix-conditioned corrector, which reranks only those K
 *      candidates with a minimal-GRU state that reads the tokens selected
 *      earlier in the block (Sec. 3.3 Eqs. 4-5; App. C.3 Eq. 9);
 *   3. left-to-right verification against the verifier distribution up to the
 *      first rejection (Sec. 3.1; Sec. 3.3; App. B Eq. 6).
 *
 * Conventions shared by every entry point:
 *  - Every tensor argument is caller-owned device memory, row-major and dense
 *    (the last dimension contiguous). The library never allocates or frees
 *    device memory; scratch lives in a caller-provided workspace of
 *    brisk_workspace_bytes() bytes and the folded corrector tables in a
 *    caller-provided buffer of brisk_tables_bytes() bytes, both 256-byte
 *    aligned. A workspace must not be shared by calls that may overlap; its
 *    contents need no initialisation.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream). Calls only enqueue work and return; results are ready when the
 *    stream reaches them. Every call may be captured into a CUDA graph.
 *  - Host-detectable problems (NULL pointers, unsupported sizes, bad modes,
 *    misaligned buffers) return an error before anything is enqueued. A
 *    failed kernel launch returns BRISK_ERR_CUDA. Problems found on the
 *    device are recorded in a status word in the workspace, read with
 *    brisk_last_device_status(); the first one of a call wins.
 *  - Logit and hidden tensors are fp32 or bf16 as the dims say; every
 *    internal sum and score is fp32. Ids are int32.
 *  - Positions are 0-based: position i of the block is the paper's i+1, and
 *    the token before position 0 is the anchor x0 (the paper's x_0).
 */
#ifndef BRISK_H
#define BRISK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum brisk_status {
  BRISK_OK = 0,
  BRISK_ERR_INVALID_ARG = 1,   /* NULL pointer, bad mode, size out of range, misaligned buffer */
  BRISK_ERR_UNSUPPORTED = 2,   /* valid request this build does not implement                   */
  BRISK_ERR_CUDA = 3,          /* a CUDA call or kernel launch failed                           */
  BRISK_ERR_TIMEOUT = 4,       /* a bounded device-side wait gave up                            */
  BRISK_ERR_NUMERIC = 5        /* a non-finite log-partition (NaN / all -inf) or a NaN score     */
} brisk_status;

typedef enum brisk_dtype { BRISK_DT_F32 = 0, BRISK_DT_BF16 = 1 } brisk_dtype;

/* Select rule of Algorithm 1(b): argmax of the refined scores (lowest rank on ties),
 * or one draw from softmax of the refined scores with a caller uniform. */
typedef enum brisk_select_mode { BRISK_SELECT_GREEDY = 0, BRISK_SELECT_SAMPLE = 1 } brisk_select_mode;

/* Verification: greedy (accept iff x_i is the verifier argmax) or speculative sampling
 * (accept iff u < min(1, p_i(x_i)/pi_i(x_i)), resample from [p_i - pi_i]_+; Sec. 3.3). */
typedef enum brisk_verify_mode { BRISK_VERIFY_GREEDY = 0, BRISK_VERIFY_STOCHASTIC = 1 } brisk_verify_mode;

/* Problem sizes. B sequences, block length L (the paper's M), vocabulary V, backbone width d,
 * K candidates, corrector width r. The corrector state has S = 2r dimensions; the position
 * embedding and the feature projection have 16 (App. C.3 head configuration, with
 * rank = hidden projection = token projection = r).
 * Limits: B >= 1; 1 <= L <= 64; 4 <= K <= 32; V >= K; d >= 8 and d % 8 == 0;
 * 16 <= r <= 512 and r % 16 == 0. */
typedef struct brisk_dims {
  int32_t B, L, V, d, K, r;
  int32_t logits_dtype;   /* brisk_dtype of logits_q / logits_p                        */
  int32_t hidden_dtype;   /* brisk_dtype of hidden, h_ctx, every weight and E_in/E_out */
} brisk_dims;

/* Corrector parameters psi and the frozen vocabulary rows (App. C.3), device pointers in
 * hidden_dtype, row-major:
 *   E_in  [V, d]   frozen input token embedding E
 *   E_out [V, d]   frozen LM-head rows E_out
 *   P_h   [r, d]   projection of MASK hidden states and of h_ctx
 *   P_e   [r, d]   projection of token embeddings
 *   P_phi [16, 5]  projection of the 5 confidence features
 *   pos   [L, 16]  position embedding
 *   W0    [S, 2r]  Init: u_0 = tanh(W0 [P_h h_ctx ; P_e E_in(x0)])
 *   Wz,Wh [S, 2r+32] minimal-GRU gate and candidate over [P_h m_i ; P_e E_in(x_{i-1}) ; pos_i ; P_phi phi_i]
 *   W_s   [r, S]   state side of the low-rank residual
 *   W_c   [r, d]   candidate side of the low-rank residual
 *   w_g   [S+5]    gate weights over [s_i ; phi_i]
 *   b_g, alpha     gate bias and gate scale: gamma_i = sigmoid(alpha) sigmoid(w_g.[s_i;phi_i] + b_g) */
typedef struct brisk_params {
  const void *E_in, *E_out;
  const void *P_h, *P_e, *P_phi, *pos;
  const void *W0, *Wz, *Wh, *W_s, *W_c, *w_g;
  float b_g, alpha;
} brisk_params;

/* Inputs and outputs of the fused tail. Output pointers marked "optional" may be NULL, in
 * which case the values are kept in the workspace only. */
typedef struct brisk_tail_io {
  const void *logits_q;     /* [B, L, V] proposal logits l^q                              */
  const void *logits_p;     /* [B, L, V] verifier logits                                  */
  const void *hidden;       /* [B, L, d] MASK hidden states m_i                           */
  const void *h_ctx;        /* [B, d]    context hidden state h_c                         */
  const int32_t *x0;        /* [B]       anchor token, the token before the block         */
  const float *u_sel;       /* [B, L] uniforms in [0,1) for sample Select (else unused)    */
  const float *u_acc;       /* [B, L] acceptance uniforms (stochastic verify)             */
  const float *u_res;       /* [B, L] residual-resampling uniforms (stochastic verify)    */
  int32_t *cand_ids;        /* optional [B, L, K] candidate ids, best first               */
  float *cand_logprob;      /* optional [B, L, K] log q_i of the candidates               */
  float *lse_q;             /* optional [B, L]    log-partition of the proposal rows      */
  int32_t *sel_tokens;      /* optional [B, L]    selected tokens x_i                     */
  float *refined;           /* optional [B, L, K] refined scores                          */
  int32_t *accepted_len;    /* [B]    accepted prefix length a, 0..L                      */
  int32_t *out_tokens;      /* [B, L] sel_tokens[0..a-1], the correction at a (if a < L), then -1 */
  int32_t *correction;      /* [B]    correction token, -1 when a == L                    */
  int32_t *next_anchor;     /* optional [B] last committed token (anchor of the next block) */
} brisk_tail_io;

/* Optional timing hooks: cudaEvent_t handles (as void*) recorded right before and right after
 * the two vocabulary-sweep kernels of brisk_decode_tail, each on the stream that kernel runs on
 * (the two launches may overlap). NULL fields are skipped. */
typedef struct brisk_events {
  void *sweep_q_begin, *sweep_q_end, *sweep_p_begin, *sweep_p_end;
} brisk_events;

/* Bytes of workspace the entry points need for `dims` (256-byte multiple). The same
 * workspace serves every entry point for these dims. 0 if dims are invalid. */
size_t brisk_workspace_bytes(const brisk_dims *dims);

/* Bytes of the folded corrector tables for `dims` (256-byte multiple); 0 if invalid. */
size_t brisk_tables_bytes(const brisk_dims *dims);

/* Fold the frozen vocabulary rows into the corrector's weights, once per weight set
 * (App. C.3: E_in, E_out and the backbone stay frozen, so P_e E_in(v), W_c E_out(v) and
 * their products with the GRU and residual matrices are fixed per token). Fills `tables`
 * (brisk_tables_bytes(dims) bytes). Must run before brisk_corrector_select /
 * brisk_decode_tail with these params; `params` buffers may be freed afterwards. */
brisk_status brisk_corrector_prepare(const brisk_dims *dims, const brisk_params *params,
                                     void *tables, void *stream);

/* Step 1 (Sec. 3.3 "C_i = TopK(q_i, K)"; App. C.3 ordered candidate set S_j): for every row
 * (b, i) of logits_q [B, L, V]: lse_q = max + log sum exp(l - max) over all V, the K ids of
 * largest logit ordered by (logit descending, id ascending) in cand_ids [B, L, K], and
 * cand_logprob = l(id) - lse_q. */
brisk_status brisk_topk_candidates(const brisk_dims *dims, const void *logits_q,
                                   int32_t *cand_ids, float *cand_logprob, float *lse_q,
                                   void *workspace, void *stream);

/* Step 1 for callers that cannot allocate device memory. The paper has no counterpart; this
 * is a deployment variant of brisk_topk_candidates with the same inputs, outputs and results
 * but no workspace argument. Some callers cannot hand the library a workspace: a plug-in that
 * runs inside another runtime and only receives its input and output buffers, an engine whose
 * memory manager owns all of HBM and forbids ad-hoc cudaMalloc, a decode loop that must not
 * allocate. This entry point keeps its scratch in a fixed 4 MiB array inside the library,
 * present on every GPU that loads the library until the process exits, and allocates nothing.
 *  - Returns BRISK_ERR_UNSUPPORTED when the problem needs more than that array holds (its
 *    per-row arrival counters and per-chunk partial results grow with B*L and K).
 *  - The first call in a CUDA context looks up the array's device address there
 *    (cudaGetSymbolAddress) and keeps it for that context; after a device reset (a new context)
 *    the next call looks it up again. Make the first call on a device before any stream capture.
 *  - Every call on a device shares the one array; calls that can overlap on the GPU (other
 *    streams, other host threads) race and must be serialised by the caller.
 *  - Device-side problems are not reported through a status word: a row without a finite
 *    logit shows as a non-finite lse_q. */
brisk_status brisk_topk_candidates_noalloc(const brisk_dims *dims, const void *logits_q,
                                           int32_t *cand_ids, float *cand_logprob, float *lse_q,
                                           void *stream);

/* Step 2 (Sec. 3.3 Eqs. 4-5; App. C.3 Eq. 9; Algorithm 1(b) loop): per sequence, sequentially
 * over positions, the minimal-GRU corrector state, the gated low-rank residual on the K
 * candidates and Select. Reads the step-1 outputs (cand_ids, cand_logprob) and logits_q
 * (for the confidence features), hidden [B, L, d], h_ctx [B, d], x0 [B]; u_sel [B, L] is
 * required for BRISK_SELECT_SAMPLE. Writes sel_tokens [B, L] and refined [B, L, K]
 * (refined_{i,k} = cand_logprob_{i,k} + gamma_i d_{i,k}). `tables` from brisk_corrector_prepare. */
brisk_status brisk_corrector_select(const brisk_dims *dims, const brisk_params *params,
                                    const void *tables, const void *hidden, const void *h_ctx,
                                    const int32_t *x0, const void *logits_q,
                                    const int32_t *cand_ids, const float *cand_logprob,
                                    int32_t select_mode, const float *u_sel,
                                    int32_t *sel_tokens, float *refined,
                                    void *workspace, void *stream);

/* Step 3 (Sec. 3.1 accept-prefix; Sec. 3.3 speculative sampling; App. B Eq. 6 strict u < alpha):
 * verifier row statistics over logits_p [B, L, V], then per sequence left to right to the first
 * rejection. Greedy: accept iff sel_tokens[b,i] is the verifier argmax (lowest id on ties); the
 * correction is that argmax. Stochastic: pi_i is softmax(refined) on cand_ids for sample Select and
 * a point mass on the selected token for greedy Select; accept iff u_acc < min(1, p/pi); at the
 * first rejection draw from the normalised [p - pi]_+ with u_res, walking ids in ascending order
 * (the verifier argmax when that mass is <= 1e-6). Writes accepted_len [B], out_tokens [B, L] and
 * correction [B]. */
brisk_status brisk_verify_block(const brisk_dims *dims, const void *logits_p,
                                const int32_t *sel_tokens, const int32_t *cand_ids,
                                const float *refined, int32_t select_mode, int32_t verify_mode,
                                const float *u_acc, const float *u_res, int32_t *accepted_len,
                                int32_t *out_tokens, int32_t *correction, void *workspace,
                                void *stream);

/* Steps 1-3 for one block step (the steps of Algorithm 1(b) after the backbone pass): the same
 * results, bit for bit, as brisk_topk_candidates + brisk_corrector_select + brisk_verify_block on
 * the same inputs. The work runs on library side streams of decreasing priority: the
 * hidden-state products; the proposal sweep, corrector and verification (the critical path);
 * the verifier-row sweep, which starts at once and fills the SMs the others leave free (this
 * applies whenever each proposal row is swept as one task: many rows, or rows too short to
 * split). When the batch is small enough that the proposal rows are swept in several chunks
 * each, the critical
 * path runs on `stream` itself: the verifier sweep starts after the proposal sweep, beside the
 * corrector; or, when both logit tensors together hold at most 64 MB, one sweep launch covers
 * the rows of both and the corrector kernel also verifies (brisk_kernels_per_tail counts the
 * launches). The call
 * only enqueues work and the results are ordered on `stream` (the side streams fork from and
 * join back to it, also under graph capture). The first call in a CUDA context creates the side
 * streams and their events: make it before any stream capture. Calls from several host threads
 * are serialised while they enqueue, and brisk_tail_graph_create holds that serialisation for
 * the whole of its capture. `ev` may be NULL.
 * logits_q and logits_p may also point to page-locked host memory (cudaHostAlloc /
 * cudaMallocHost, or cudaHostRegister with cudaHostRegisterMapped; mapped into the device's
 * unified address space): the kernels then read the logits in place over the host link, with
 * the same results bit for bit (about 210 GB/s on a GB300 with its Grace host, the rate of a
 * copy-engine copy of the same buffers, without the copy's second pass through HBM). Every
 * other pointer is device memory; memory that is neither is undefined behaviour. */
brisk_status brisk_decode_tail(const brisk_dims *dims, const brisk_params *params,
                               const void *tables, const brisk_tail_io *io, int32_t select_mode,
                               int32_t verify_mode, void *workspace, const brisk_events *ev,
                               void *stream);

/* ---- The decode tail as a replayable CUDA graph (App. F: fused head plus CUDA Graph replay) ----
 *
 * brisk_tail_graph_create makes one direct brisk_decode_tail call with these arguments (it
 * checks them and prepares the library's side streams), then captures a second call on
 * `stream` (a non-default stream, thread-local capture) into a graph whose launches read and
 * write exactly the buffers of `io`, `tables` and `workspace`. brisk_tail_graph_launch replays
 * it on `stream`: refresh the inputs in place between launches; with io->x0 == io->next_anchor
 * the anchor of block t+1 is the last committed token of block t, on the device. The buffers
 * must outlive the graph; the graph and the workspace must not be used by overlapping launches.
 * Returns the status of the direct call, BRISK_ERR_INVALID_ARG for a NULL out/stream, or
 * BRISK_ERR_CUDA if capture or instantiation fails. */
typedef struct brisk_graph brisk_graph;
brisk_status brisk_tail_graph_create(const brisk_dims *dims, const brisk_params *params,
                                     const void *tables, const brisk_tail_io *io,
                                     int32_t select_mode, int32_t verify_mode, void *workspace,
                                     void *stream, brisk_graph **out);
brisk_status brisk_tail_graph_launch(brisk_graph *graph, void *stream);
void brisk_tail_graph_destroy(brisk_graph *graph);

/* Kernels one brisk_decode_tail call launches for `dims` (0 if dims are invalid). */
int32_t brisk_kernels_per_tail(const brisk_dims *dims);

/* Reads the device status word of `workspace` (synchronises `stream`): BRISK_OK or the first
 * device-side problem recorded by the most recent call on this workspace (every call clears the
 * word when it starts). Device-side problems: a non-finite log-partition or a candidate id that
 * a row with no finite logit left out of range, or a NaN refined score (BRISK_ERR_NUMERIC; Select
 * then ranks NaN below every number, so the selection is still a candidate); an anchor or selected token
 * outside [0, V) (BRISK_ERR_INVALID_ARG; the id is replaced by 0 so that nothing reads out of
 * bounds). With clear != 0 the word is reset to BRISK_OK afterwards. */
brisk_status brisk_last_device_status(void *workspace, int32_t clear, void *stream);

/* Sets the limit, in SM clock cycles, of the bounded device-side waits (the tensor-core
 * products' pipeline and accumulator waits, which no other kernel has: the sweep, corrector and
 * verification kernels never wait on another CTA or on a copy). cycles <= 0 restores the default
 * of 4e9 cycles (about 2 s). Returns the previous limit. The value is read when a launch is
 * enqueued and passed to the kernel (a captured graph keeps the value it was captured with); it
 * is process-wide. When a wait gives up, the call records BRISK_ERR_TIMEOUT in the device status,
 * its outputs are undefined, and the kernel still waits (up to the default limit) for the copies
 * and tensor-core operations it started before it frees its resources and returns, so the CUDA
 * context stays usable. A short limit makes waits give up while their data is still arriving:
 * tests of the failure path use it. No counterpart in the paper (failure detection). */
int64_t brisk_set_wait_limit(int64_t cycles);

/* Human-readable name of a status code (static storage). */
const char *brisk_status_string(brisk_status status);

/* ---- Acceptance profile and risk-reward position weights (Sec. 2.2; Sec. 3.2 Eqs. 2-3) ----
 *
 * The paper estimates the per-position acceptance a_i of a verified block as one minus the
 * rejection rate at position i among the blocks whose verification reached i, and turns the
 * profile into tokens per forward (TPF) and position weights for the proposal loss. */

/* Adds one block step's accepted lengths to running counts (device): for every position
 * i < L, counts[i] += #{b : accepted_len[b] >= i} (blocks that reached i) and
 * counts[L + i] += #{b : accepted_len[b] >= i + 1} (blocks that accepted i). accepted_len
 * [B] int32 (device, values in 0..L, the output of brisk_verify_block / brisk_decode_tail);
 * counts [2L] uint64 (device, caller-owned, zeroed by the caller before the first step).
 * Integer sums: the counts do not depend on timing. Lengths outside 0..L are clamped.
 * 1 <= L <= 64, B >= 0. */
brisk_status brisk_acceptance_counts(const int32_t *accepted_len, int32_t B, int32_t L,
                                     unsigned long long *counts, void *stream);

/* Host-side (no device work). For a profile a[0..M-1] (a_i in [0, 1], position i of the block)
 * and per-length committed tokens g[0..M] and forward costs c[0..M] (Eq. 2), writes
 * tpf = sum_k Pr(L=k) g_k / sum_k Pr(L=k) c_k with Pr(L=k) = A_k (1 - a_k) for k < M and A_M
 * for k = M (A_k = a_0 ... a_{k-1}); w_raw[i] = -dFPT/dz_i with FPT = 1/TPF and
 * z_i = log(a_i / (1 - a_i)); w_bar[i] = M w_raw[i] / (sum_j w_raw[j] + eps) (Eq. 3). g or c
 * NULL means g_k = k + 1 and c_k = 1 (one guaranteed token, unit cost: TPF = 1 + sum A_k).
 * Any output pointer may be NULL. 1 <= M <= 64; BRISK_ERR_INVALID_ARG for a NULL profile, an
 * a_i outside [0, 1] or a zero expected cost. */
brisk_status brisk_acceptance_weights(int32_t M, const double *a, const double *g, const double *c,
                                      double eps, double *tpf, double *w_raw, double *w_bar);

/* ---- Same-state replay diagnostics (App. B, "Same-state replay", Eq. 6) ----
 *
 * Runs the candidates, the verifier rows' log-partition and the corrector with the head
 * conditioned on the factual base prefix (the token fed forward at every position is the base
 * selection: the Select rule applied to the base scores log q with the same draw u_sel, i.e.
 * rank 0 under greedy selection), then scores the base token and the head's token of every
 * position under one shared draw: alpha_i(x) = min(1, p_i(x) / q_i(x)) with q_i the proposal
 * normalised over the full vocabulary and p_i the verifier, J_i(x) = [u_acc_i < alpha_i(x)].
 * Inputs as brisk_corrector_select plus logits_p [B, L, V] and u_acc [B, L] f32 (device).
 * Outputs (device): head_tokens [B, L] int32; flags [B, L] int32 with bit 0 = J(base),
 * bit 1 = J(head), bit 2 = first breaker (the first position whose base token the draw
 * rejects), bit 3 = intervention (head token != base token), bit 4 = rescue (J(base) = 0 and
 * J(head) = 1 at the first breaker), bit 5 = regression (J(head) = 0 at a position before the
 * first breaker, where J(base) = 1); first_breaker [B] int32 (L if none); refined [B, L, K]
 * f32 or NULL. */
brisk_status brisk_replay_diagnostics(const brisk_dims *dims, const brisk_params *params,
                                      const void *tables, const void *hidden, const void *h_ctx,
                                      const int32_t *x0, const void *logits_q,
                                      const void *logits_p, int32_t select_mode,
                                      const float *u_sel, const float *u_acc,
                                      int32_t *head_tokens, int32_t *flags,
                                      int32_t *first_breaker, float *refined, void *workspace,
                                      void *stream);

/* ---- Distillation loss of the refinement head (App. C.3, Eq. 10) ----
 *
 * The training objective of the corrector on a batch of blocks: at every reached position j
 * (j <= min(accepted_len[b], L-1): the accepted prefix and the first rejected position),
 * CE(p_S, r) + beta KL(q_S || r), where p_S = the verifier distribution restricted to the K
 * candidates of position j and renormalised (from logits_p at cand_ids), q_S = the proposal
 * distribution restricted to them (from cand_logprob), r = softmax(refined); the loss is one
 * mean over all reached positions of the batch (the paper uses beta = 0.01).
 * logits_p [B, L, V] (dims.logits_dtype), cand_ids / cand_logprob / refined [B, L, K],
 * accepted_len [B] int32 (values outside 0..L are clamped), all device. Writes loss [1] f32
 * (device) and, unless grad_refined is NULL, d loss / d refined [B, L, K] f32 (device; zero at
 * unreached positions). The loss does not depend on timing. An out-of-range candidate id is
 * replaced by 0 and reported as BRISK_ERR_INVALID_ARG in the device status. */
brisk_status brisk_distill_loss(const brisk_dims *dims, const void *logits_p,
                                const int32_t *cand_ids, const float *cand_logprob,
                                const float *refined, const int32_t *accepted_len, float beta,
                                float *loss, float *grad_refined, void *workspace, void *stream);

/* Host-side: the gains and costs that make Eq. 2 the ISD instantiation the paper uses for FPT
 * and the weights (App. C.1, Eq. 8: TPF = (2 + sum_{k=1}^{M-1} A_k) / (2 - A_M), M = N - 1):
 * g[k] = 2 + min(k, M - 1) and c[k] = 2 for k < M, c[M] = 1, written for k = 0..M (M + 1 values
 * each, caller-owned host arrays), to pass to brisk_acceptance_weights. BRISK_ERR_INVALID_ARG
 * for M outside 1..64 or a NULL array. */
brisk_status brisk_isd_costs(int32_t M, double *g, double *c);

/* Host-side: tokens per forward of the ISD stride-N rule at constant rejection r (Sec. 2.2):
 * (2 + sum_{i=1}^{N-2} (1-r)^i) / (2 - (1-r)^{N-1}); NaN for N < 2 or r outside [0, 1]. */
double brisk_tpf_isd(int32_t N, double r);

#ifdef __cplusplus
}
#endif

#endif /* BRISK_H */
