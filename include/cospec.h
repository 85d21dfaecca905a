/*
 * cospec.h -- C ABI of the GB300 (sm_103a) verify/arbitrate round of
 * collaborative speculative decoding (CoSpec).
 *
 * One round (Sec. 3.1 and Sec. 3.3 of the paper; App. F, Inference Procedure):
 *   1. cospec_verify_attn            per layer: attention of the K+1 block rows
 *                                    over a paged bf16 KV cache (Eq. 2)
 *   2. cospec_lmhead_argmax_features LM head fused with argmax and the
 *                                    log-prob statistics (Eq. 2, Eq. 23)
 *   3. cospec_arbitrate              accept/reject at every draft/target
 *                                    mismatch (Eq. 3, Eq. 13-14, Eq. 17)
 *   4. cospec_accept_commit          accepted length and emitted tokens
 *                                    (Eq. 15), KV commit of the accepted rows
 *
 * Conventions shared by every call
 *  - Every array pointer is a DEVICE pointer owned by the caller; the library
 *    allocates nothing, frees nothing and never synchronises the stream,
 *    except cospec_get_device_error.  `stream` is a cudaStream_t (NULL = the
 *    legacy default stream).  All calls are asynchronous.
 *  - bf16 tensors are passed as uint16_t bit patterns, row-major, innermost
 *    dimension last, densely packed.
 *  - Host-side argument checks run before anything is launched; a failing
 *    check returns a negative cospec_status and launches nothing.
 *  - Data-dependent violations found on the device (a page id outside the
 *    pool, a context that does not fit its page-table row, a token id outside
 *    the vocabulary, a pipeline wait that timed out) skip the offending unit
 *    and set a bit in a device error word (COSPEC_DEVERR_*), which
 *    cospec_get_device_error reads and clears.  No kernel traps.
 *  - Calls may come from any host thread and several threads at once; each
 *    works on the calling thread's current device (its primary context is
 *    made current on the thread's first call).  Calls that share a device
 *    error word or the no-allocation LM-head scratch on one device see each
 *    other's contents there.
 *  - Block geometry: a round verifies R = K + 1 rows per sequence.  Row 0 is
 *    the last token emitted by the previous round (its KV is not committed
 *    yet), rows 1..K are the draft tokens y_hat_1..y_hat_K.  Row j sits at
 *    absolute position ctx_len[b] + j and its LM-head row predicts
 *    y_tilde_{j+1}.
 */
#ifndef COSPEC_H
#define COSPEC_H

#include <stddef.h>
#include <stdint.h>

#if defined(_WIN32)
#define COSPEC_API
#else
#define COSPEC_API __attribute__((visibility("default")))
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  COSPEC_OK = 0,
  COSPEC_ERR_INVALID_ARG = -1,  /* null pointer, bad size or inconsistent shape */
  COSPEC_ERR_UNSUPPORTED = -2,  /* valid but outside the shapes the kernels handle */
  COSPEC_ERR_WORKSPACE = -3,    /* workspace missing or smaller than required */
  COSPEC_ERR_CUDA = -4,         /* a CUDA runtime call or a launch failed */
  COSPEC_ERR_DEVICE_CHECK = -5  /* the device error word was non-zero */
} cospec_status;

/* Bits of the device error word. */
#define COSPEC_DEVERR_PAGE 1     /* page id outside [0, num_pages) */
#define COSPEC_DEVERR_CTX 2      /* ctx_len < 0 or ctx_len > max_pages_per_seq * page_size
                                    (attention), or ctx_len plus the accepted rows >
                                    max_pages_per_seq * page_size (commit) */
#define COSPEC_DEVERR_TOKEN 4    /* token id outside the vocabulary */
#define COSPEC_DEVERR_TIMEOUT 8  /* a bounded pipeline wait gave up (never expected) */
#define COSPEC_DEVERR_OFFSETS 16 /* a group / round offset array is not non-decreasing within
                                    its range (RL call); the group is skipped */

/* Human-readable name of a cospec_status value (static string). */
COSPEC_API const char* cospec_status_string(int status);

/* Name of the CUDA runtime error behind the last COSPEC_ERR_CUDA that a call
 * made on this host thread returned ("cudaSuccess" when there was none;
 * static string).  Lets a caller tell, e.g., an invalid stream from an
 * unsupported launch configuration. */
COSPEC_API const char* cospec_last_cuda_error(void);

/* Reads the device error word into *flags, then clears it.  Synchronises
 * `stream` first, so every kernel queued before is included.  Returns
 * COSPEC_OK, or COSPEC_ERR_DEVICE_CHECK when *flags != 0. */
COSPEC_API int cospec_get_device_error(int* flags, void* stream);

/* Number of SMs of the current device (used to size grids; cached). */
COSPEC_API int cospec_num_sms(void);

/* ------------------------------------------------------------------------ */
/* 1. Verify attention (Sec. 3.1, Eq. 2: one teacher-forced pass of the
 *    target over [x, y^(<r), y_hat_1..y_hat_K]; this call is the attention
 *    of one layer of that pass for the K+1 rightmost positions).
 *
 *    For sequence b, query head h, block row j:
 *      o = softmax(q . k^T * softmax_scale + mask) . v
 *    over the ctx_len[b] committed positions of the paged cache followed by
 *    block rows 0..j of (k_blk, v_blk) (causal inside the block).  Query
 *    head h reads KV head h / (num_q_heads / num_kv_heads) (GQA).
 *
 *    q        bf16 [batch, rows, num_q_heads, head_dim]
 *    k_blk    bf16 [batch, rows, num_kv_heads, head_dim]   this layer's block keys
 *    v_blk    bf16 [batch, rows, num_kv_heads, head_dim]
 *    k_pages  bf16 [num_pages, num_kv_heads, page_size, head_dim]   this layer's pool
 *    v_pages  bf16 [num_pages, num_kv_heads, page_size, head_dim]
 *    page_table int32 [batch, max_pages_per_seq]: logical page p of sequence b
 *             is physical page page_table[b * max_pages_per_seq + p]; only the
 *             first ceil(ctx_len[b] / page_size) entries are read.
 *    ctx_len  int32 [batch]
 *    out      bf16 [batch, rows, num_q_heads, head_dim] (may not alias inputs)
 *    max_ctx  the expected largest ctx_len[*] (host-side; 0 <= max_ctx <=
 *             max_pages_per_seq * page_size).  It only sizes the KV split: a
 *             context above it is still attended in full and correctly, only
 *             with a split planned for a shorter one; it sets no error bit.
 *    No workspace: the KV range of a (sequence, KV head) is split over the
 *    CTAs of one thread-block cluster, whose partial results merge in
 *    distributed shared memory.  Two kernels implement the call: one on
 *    mma.sync tensor-core tiles, and one on tcgen05 (TMEM accumulators, the
 *    query rows as the MMA M dimension, up to 128 rows of a KV head per
 *    CTA), used when a KV head has more than 32 query rows (and at most 64
 *    query heads share the KV head).  Batches of up to 64 sequences are
 *    processed longest context first; larger ones in index order (a caller
 *    can order them).
 *    Supported: head_dim in {64, 128}; page_size == 16; rows <= 64;
 *    num_q_heads % num_kv_heads == 0; (num_q_heads / num_kv_heads) * rows <= 512.
 * ------------------------------------------------------------------------ */
typedef struct {
  int batch;
  int rows;              /* R = K + 1 */
  int num_q_heads;
  int num_kv_heads;
  int head_dim;
  int page_size;
  int max_pages_per_seq;
  int num_pages;
  float softmax_scale;   /* <= 0 selects 1/sqrt(head_dim) */
  int flags;             /* COSPEC_ATTN_* bits, 0 by default */
} cospec_attn_dims;

/* The call may start reading ctx_len, page_table and the cached pages before
 * the kernel queued just before it on the stream has finished: set it only
 * when that kernel writes none of them (e.g. between the layers of one
 * round, where only q / k_blk / v_blk come from the previous layer). */
#define COSPEC_ATTN_KV_STABLE 1

/* Every block row attends to every block row instead of rows 0..j only: the
 * draft/target region of the arbitrator's input (Sec. 3.3), which sees the
 * whole context causally cached before it and itself bidirectionally, the
 * context never seeing the region.  With the region's 2K+3 tokens as the
 * block (rows <= 64, i.e. K <= 30) this is the arbitrator LM's attention
 * for one round. */
#define COSPEC_ATTN_BLOCK_FULL 2

/* Launch plan cospec_verify_attn would use for these dimensions (flags
 * included: a small batch launched with COSPEC_ATTN_KV_STABLE, which may
 * overlap the kernel before it, can take a larger KV split than one that
 * starts on an idle GPU) on the current device: *kernel = 0 (mma.sync) or 1
 * (tcgen05), *splits = CTAs per (sequence, KV head, row group), 1 to 16.
 * Host only; returns COSPEC_OK or the error cospec_verify_attn would return
 * for the dimensions. */
COSPEC_API int cospec_verify_attn_plan(const cospec_attn_dims* dims, int max_ctx, int* kernel,
                                       int* splits);

/* Residency model for cospec_verify_attn_plan_model: how many clusters of
 * `splits` CTAs of one attention kernel variant a device keeps resident at
 * once (0: such a cluster cannot be scheduled).  kernel 0 (mma.sync):
 * `rows` = padded query rows of a CTA (16, 32 or 64), `block_rows` = the
 * block's keys padded to 16; kernel 1 (tcgen05): `rows` = 128 (the query
 * rows of a CTA), `block_rows` as for kernel 0. */
typedef long long (*cospec_resident_fn)(int kernel, int rows, int block_rows, int splits,
                                        void* user);

/* The plan cospec_verify_attn_plan computes, for a device described by its
 * SM count and a residency model instead of the current device (the same
 * rules: kernel choice, KV split, one wave of resident clusters for small
 * batches).  Host only, no CUDA call: it lets a host without a GPU check or
 * predict the plan for any machine.  Errors as for cospec_verify_attn_plan,
 * and COSPEC_ERR_INVALID_ARG for num_sms < 1 or a null model. */
COSPEC_API int cospec_verify_attn_plan_model(const cospec_attn_dims* dims, int max_ctx,
                                             int num_sms, cospec_resident_fn resident, void* user,
                                             int* kernel, int* splits);

COSPEC_API int cospec_verify_attn(const cospec_attn_dims* dims, int max_ctx,
                                  const uint16_t* q, const uint16_t* k_blk, const uint16_t* v_blk,
                                  const uint16_t* k_pages, const uint16_t* v_pages,
                                  const int32_t* page_table, const int32_t* ctx_len,
                                  uint16_t* out, void* stream);

/* ------------------------------------------------------------------------ */
/* 2. LM head fused with argmax and log-prob statistics (Eq. 2 gives the
 *    target prediction y_tilde = argmax of each row's logits; Eq. 23 defines
 *    l_i = log p_T(y_hat_i | prefix) = x[y_hat_i] - lse).
 *
 *    For each of the M rows: x = hidden[m] . W^T (fp32 accumulation of bf16
 *    products; the M x V logits are never written to memory) and
 *      argmax[m]   = lowest id among the maximal logits (y_tilde)
 *      stats[m][0] = max_v x_v
 *      stats[m][1] = largest logit over ids != argmax (equals [0] on a tie)
 *      stats[m][2] = lse = log sum_v exp(x_v)
 *      stats[m][3] = entropy = lse - sum_v softmax(x)_v x_v
 *      stats[m][4] = x[draft_for_row[m]], NaN when draft_for_row[m] == -1
 *
 *    hidden   bf16 [M, d];  w  bf16 [V, d] (nn.Linear weight layout)
 *    draft_for_row int32 [M] in [-1, V): the draft id scored by row m
 *    argmax   int32 [M];  stats float32 [M, 5]
 *    ws       >= cospec_lmhead_workspace(M, d, V) bytes (no initialisation)
 *    Supported: d % 64 == 0, 1 <= M, V >= 1; hidden and w 16-byte aligned.
 *    Runs on tcgen05 tensor cores (TMEM accumulators, TMA-fed operands).
 * ------------------------------------------------------------------------ */
COSPEC_API size_t cospec_lmhead_workspace(int M, int d, int V);
COSPEC_API int cospec_lmhead_argmax_features(int M, int d, int V, const uint16_t* hidden,
                                             const uint16_t* w, const int32_t* draft_for_row,
                                             int32_t* argmax, float* stats, void* ws,
                                             size_t ws_bytes, void* stream);

/* Stochastic decoding (Sec. 3.1 "Stochastic decoding"; App. C.3 draws the
 * draft and target candidates at temperature T = 1 and arbitrates between
 * the pair exactly as in greedy decoding).  Same contraction, statistics and
 * workspace as cospec_lmhead_argmax_features, but the target candidate
 * written to sample[m] is a draw from softmax(x / T) instead of the argmax:
 *
 *   sample[m] = argmax_v ( x_v / T + g_{m,v} ),  g = -log(-log u)   (Gumbel-max)
 *   u_{m,v}   = (floor(r / 2^9) + 0.5) / 2^23,  r = output (m mod 4) of
 *               Philox4x32-10 at counter (v, floor(m / 4), 0, 0) under the
 *               key (seed mod 2^32, floor(seed / 2^32))
 *
 * (Salmon et al., SC 2011), ties going to the lowest id.  stats[m][*] are
 * the statistics of the logits x themselves, as in the greedy call.
 *
 *    temperature > 0 and finite (1 for the paper's stochastic setting).
 *    seed      DEVICE pointer to one uint64 (8-byte aligned), read when the
 *              kernel runs, so a captured graph draws fresh noise whenever
 *              the caller rewrites it between replays.
 *    sample    int32 [M];  other arguments as for the greedy call.
 * This is not distribution-preserving speculative sampling: the paper's
 * method uses the sampled pair as two candidates for arbitration. */
COSPEC_API int cospec_lmhead_sample_features(int M, int d, int V, const uint16_t* hidden,
                                             const uint16_t* w, const int32_t* draft_for_row,
                                             float temperature, const uint64_t* seed,
                                             int32_t* sample, float* stats, void* ws,
                                             size_t ws_bytes, void* stream);

/* The LM head for speculative sampling at temperature T (the exact-match
 * baseline of Sec. 3.1 "Stochastic decoding" / App. C.3, see
 * cospec_sps_accept): the scaled logits x / T are written out, and the
 * statistics are those of x / T.
 *
 *    logits   float32 [M, V]: logits[m][v] = (hidden[m] . W[v]) / T (4-byte aligned)
 *    argmax   int32 [M]: lowest id among the maximal logits (as the greedy call)
 *    stats    float32 [M, 5]: as the greedy call, for the scaled logits x / T
 *             (stats[m][2] = log sum_v exp(x_v / T); stats[m][4] = x[draft] / T)
 *    temperature > 0 and finite; other arguments and the workspace as for
 *    cospec_lmhead_argmax_features.
 * The M x V logits are written to memory (M * V * 4 bytes); the greedy and
 * sampling calls never write them. */
COSPEC_API int cospec_lmhead_logits_features(int M, int d, int V, const uint16_t* hidden,
                                             const uint16_t* w, const int32_t* draft_for_row,
                                             float temperature, int32_t* argmax, float* stats,
                                             float* logits, void* ws, size_t ws_bytes,
                                             void* stream);

/* Same computation and outputs as cospec_lmhead_argmax_features, for callers
 * that cannot allocate device memory or hand this library a workspace -- for
 * example a serving engine that reserves nearly all HBM for its KV cache and
 * allows no allocation while decoding, or a plug-in inside a framework that
 * owns the device's memory.  (The paper has no counterpart; this is an
 * interface convenience of this library.)
 *
 * The per-CTA partial statistics go to a fixed 1.25 MiB scratch array
 * compiled into the library, present on every GPU that loads it until the
 * process exits; nothing is allocated and nothing needs clearing, since each
 * call overwrites the scratch it reads.  The first call on each device looks
 * up the scratch's device address (cudaGetSymbolAddress); make that first
 * call before any stream capture.  All calls share the one array, so calls
 * whose execution overlaps on the GPU (other streams, other host threads)
 * race and give wrong results: keep them ordered on one stream.
 * Limits: M <= 512 rows per call and at most 256 persistent CTAs (SMs);
 * larger requests return COSPEC_ERR_UNSUPPORTED. */
COSPEC_API int cospec_lmhead_argmax_features_noalloc(int M, int d, int V, const uint16_t* hidden,
                                                     const uint16_t* w,
                                                     const int32_t* draft_for_row,
                                                     int32_t* argmax, float* stats, void* stream);

/* ------------------------------------------------------------------------ */
/* 2b. Speculative-sampling acceptance: the distribution-preserving baseline
 *    that the paper compares against at T = 1 (Sec. 3.1 "Stochastic
 *    decoding"; App. C.3: standard speculative sampling with acceptance-ratio
 *    correction, Leviathan et al. 2023 / Chen et al. 2023).  It replaces the
 *    arbitration step of a CoSpec round.
 *
 *    With p_i = softmax(x_{i-1} / T) (block row i-1's scaled logits) and the
 *    draft's distribution q_i at draft position i:
 *      ratio[b][i-1] = min(1, p_i(y_hat_i) / q_i(y_hat_i))   (1 when q_i(y_hat_i) = 0)
 *      y_hat_i is accepted iff u * q_i(y_hat_i) < p_i(y_hat_i), u the uniform of
 *        (b, i): output word 0 of Philox4x32-10 at counter (i - 1, b, 1, 0)
 *        under the key (seed mod 2^32, floor(seed / 2^32)),
 *        u = (floor(r / 2^9) + 0.5) / 2^23;
 *      at the first rejection i*, target[b][i*-1] = a draw from
 *        max(0, p_{i*} - q_{i*}) (renormalised); with no rejection,
 *        target[b][K] = a draw from p_{K+1}.  Both draws are Gumbel-max,
 *        argmax_v (log w(v) + g_{m,v}), with the Gumbel noise of block row
 *        m = b (K + 1) + row that cospec_lmhead_sample_features uses (a
 *        residual with no positive entry, possible only through rounding,
 *        falls back to p).
 *    accept[b][i-1] = 1 before the stop row, 0 from it on; target[b][j] =
 *    y_hat_{j+1} before the stop row, -1 after it.  Passing (target, accept)
 *    as (argmax, accept) to cospec_accept_commit then yields the accepted
 *    length, the emitted tokens and the KV commit.
 *
 *    draft  int32 [B, K]
 *    stats  float32 [B*(K+1), 5] and logits float32 [B*(K+1), V] from
 *           cospec_lmhead_logits_features at temperature T
 *    q      float32 [B, K, V]: the draft's distribution at every position
 *    seed   DEVICE pointer to one uint64 (8-byte aligned), read when the kernel runs
 *    target int32 [B, K+1]; accept uint8 [B, K]; ratio float32 [B, K]
 *    ws     >= cospec_sps_workspace(B) bytes, 16-byte aligned (no initialisation)
 *    Supported: 0 <= K <= 31 (draft, q, accept, ratio may be NULL when K = 0).
 *    A draft id outside [0, V) sets COSPEC_DEVERR_TOKEN and is rejected. */
COSPEC_API size_t cospec_sps_workspace(int B);
COSPEC_API int cospec_sps_accept(int B, int K, int V, const int32_t* draft, const float* stats,
                                 const float* logits, const float* q, const uint64_t* seed,
                                 int32_t* target, uint8_t* accept, float* ratio, void* ws,
                                 size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------ */
/* 3. Arbitration at draft/target mismatches (Sec. 3.3).
 *
 *    Delta_i = 1[draft[b,i-1] == argmax[b,i-1]] (Eq. 3).  Matches are forced
 *    accepted: p = sigma(+inf) = 1, accept = 1 (Eq. 13-14).  At a mismatch
 *    p = sigma(z) with z = w2 . ReLU(W1 f_i + b1) + b2 for policy_mode 0,
 *    p = 0 for policy_mode 1 ("always target", exact-match decoding) and
 *    p = 1 for policy_mode 2 ("always draft"); accept = 1[p > lambda]
 *    (Eq. 17, strict).  f_i is the 8-feature vector built from the target
 *    statistics of rows i-1 and i (F0 = x_{i-1}[y_hat_i] - lse_{i-1},
 *    F1 = max_{i-1} - lse_{i-1}, F2 = max_{i-1} - second_{i-1},
 *    F3 = entropy_{i-1}, F4 = max_i - lse_i, F5 = x_i[y_hat_{i+1}] - lse_i
 *    (0 at i = K), F6 = i/K, F7 = #{j < i : Delta_j = 1}/K).
 *
 *    draft  int32 [B, K];  argmax int32 [B, K+1];  stats float32 [B, K+1, 5]
 *    w1 float32 [mlp_hidden, 8], b1 [mlp_hidden], w2 [mlp_hidden] (device;
 *    may be NULL when policy_mode != 0);  p_out float32 [B, K];
 *    accept uint8 [B, K].  Supported: 0 <= K <= 31, mlp_hidden <= 1024.
 * ------------------------------------------------------------------------ */
#define COSPEC_POLICY_MLP 0
#define COSPEC_POLICY_TARGET 1
#define COSPEC_POLICY_DRAFT 2

COSPEC_API int cospec_arbitrate(int B, int K, const int32_t* draft, const int32_t* argmax,
                                const float* stats, int mlp_hidden, const float* w1,
                                const float* b1, const float* w2, float b2, float lambda,
                                int policy_mode, float* p_out, uint8_t* accept, void* stream);

/* ------------------------------------------------------------------------ */
/* 4. Accepted length, emitted tokens and KV commit (Eq. 15; App. F).
 *
 *    s_b = min{i : Delta_i = 0 and accept_i = 0}, else K+1.  The round emits
 *    draft_1..draft_{s-1} followed by argmax row s-1 (y_tilde_s; the bonus
 *    when s = K+1).  Block rows 0..s-1 of every layer's staging K/V are then
 *    copied to cache positions ctx_len[b] .. ctx_len[b]+s-1 through the page
 *    table, and ctx_len[b] += s.  Rows after s never reach the cache.
 *
 *    draft int32 [B, K]; argmax int32 [B, K+1]; accept uint8 [B, K]
 *    k_blk, v_blk  bf16 [num_layers, B, K+1, num_kv_heads, head_dim]
 *    k_pages, v_pages  bf16: layer l's pool [num_pages, num_kv_heads,
 *             page_size, head_dim] starts pool_layer_stride elements after
 *             layer l-1's.  With num_layers > 1, pool_layer_stride must be
 *             >= num_pages*Hkv*P*D (layers never share cells; 0 or a smaller
 *             stride returns COSPEC_ERR_INVALID_ARG); with num_layers == 1 it
 *             is ignored.  A pool that stands for several layers at once is
 *             committed with num_layers = 1 and one layer's staging rows.
 *    dims     the attention geometry (batch == B, rows == K+1)
 *    ctx_len  int32 [B], updated in place
 *    accept_len int32 [B]; emitted int32 [B, K+1] (padded with -1)
 * ------------------------------------------------------------------------ */
COSPEC_API int cospec_accept_commit(int B, int K, int num_layers, const cospec_attn_dims* dims,
                                    const int32_t* draft, const int32_t* argmax,
                                    const uint8_t* accept, const uint16_t* k_blk,
                                    const uint16_t* v_blk, uint16_t* k_pages, uint16_t* v_pages,
                                    long long pool_layer_stride, const int32_t* page_table,
                                    int32_t* ctx_len, int32_t* accept_len, int32_t* emitted,
                                    void* stream);

/* ------------------------------------------------------------------------ */
/* 5. RL stage: reward shaping, returns and advantages (Sec. 3.4).
 *
 *    A batch of prompt groups: group x owns rollouts group_off[x] ..
 *    group_off[x+1]-1, rollout m owns rounds round_off[m] .. round_off[m+1]-1,
 *    and round r holds K draft positions (index i-1 for position i): match
 *    (Delta_i, Eq. 3), accept (a_i; ignored at matches) and ell
 *    (log p_T(y_hat_i | ...), Eq. 23).  Per round: s = first rejected
 *    mismatch else K+1, i* = first mismatch, rho = (s - i*) / (K+1 - i*), the
 *    effective decisions I_r = mismatches at positions <= min(s, K).
 *      g      correct rollout: rho; incorrect: -alpha |ell_i| for accepted
 *             mismatches before the first rejection, -beta at the rejection
 *      J[m]   sum of g over the rollout's effective decisions
 *      Jbar   J, with the correct rollouts of a mixed group scaled by
 *             gamma = sum_incorrect |J| / (sum_correct J + eps)
 *      adv[m] eta (Jbar - mu) / (sigma + eps) over the group (population
 *             sigma; eta = eta_fail for all-incorrect groups, else 1)
 *      adv_dec  correct: rho * adv[m]; incorrect: |g| / sum |g| * adv[m]
 *    With ratio, p_new, p_ref (pi_theta / pi_old for the taken action,
 *    pi_theta(a=1), pi_ref(a=1) per decision) also the objective:
 *      loss[0] = sum min(ratio A, clip(ratio, 1 -+ clip_eps) A), loss[1] =
 *      sum Bernoulli entropy of p_new, loss[2] = sum KL(p_new || p_ref) over
 *      the effective decisions, loss[3] = -loss[0] - beta_h loss[1] + beta_kl loss[2].
 *
 *    group_off int32 [num_groups+1]; correct uint8 [num_rollouts];
 *    round_off int32 [num_rollouts+1]; match, accept uint8 [num_rounds, K];
 *    ell float32 [num_rounds, K]; 1 <= K <= 64.
 *    Outputs (float32): g, adv_dec [num_rounds, K] (0 outside effective
 *    decisions), eff uint8 [num_rounds, K], rho [num_rounds] (NaN without a
 *    mismatch), J, Jbar, adv [num_rollouts]; loss [4] (only when ratio,
 *    p_new and p_ref are given; all three or none).  Group statistics are
 *    computed in float64.  ws >= cospec_rl_workspace(...) bytes.
 * ------------------------------------------------------------------------ */
typedef struct {
  float alpha;     /* risk penalty weight (the paper: 1.0) */
  float beta;      /* rejection penalty (0.25) */
  float eta_fail;  /* weight of all-incorrect groups (0.5) */
  float eps;       /* normaliser epsilon, > 0 */
  float clip_eps;  /* PPO clip range (0.2) */
  float beta_h;    /* entropy coefficient (0.01) */
  float beta_kl;   /* KL coefficient (0.02) */
} cospec_rl_params;

COSPEC_API size_t cospec_rl_workspace(int num_groups, int num_rollouts);
COSPEC_API int cospec_rl_advantages(int num_groups, int num_rollouts, int num_rounds, int K,
                                    const int32_t* group_off, const uint8_t* correct,
                                    const int32_t* round_off, const uint8_t* match,
                                    const uint8_t* accept, const float* ell,
                                    const cospec_rl_params* params, const float* ratio,
                                    const float* p_new, const float* p_ref, float* g,
                                    uint8_t* eff, float* rho, float* J, float* Jbar, float* adv,
                                    float* adv_dec, float* loss, void* ws, size_t ws_bytes,
                                    void* stream);

#ifdef __cplusplus
}
#endif

#endif /* COSPEC_H */
