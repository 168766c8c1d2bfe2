/*
 * tgvkv.h -- C ABI of the TGV-KV eviction step on one GB300 (sm_103a).
 *
 * TGV-KV ("Text-Grounded KV Eviction for Vision-Language Models") runs once per
 * request after the prefill (Section 1; Section 3.3).  Given, for every layer,
 * the cached keys/values and the queries of the text tokens, it
 *   1. scores every vision key by text-weighted attention (TWR, Eq. 6-8),
 *   2. turns each layer's text-vision attention sum into a layer budget
 *      (TVB, Eq. 5 with x = TV),
 *   3. keeps all text KV and the top-scoring vision KV of each head
 *      (TPR, Eq. 10, case b_l > N_t), and
 *   4. gathers the survivors into a compacted, variable-length cache.
 * The four steps are the four calls tgvkv_score, tgvkv_budget, tgvkv_select
 * and tgvkv_compact; tgvkv_evict runs all of them in one call.
 *
 * Conventions shared by every call
 * --------------------------------
 * - Every data pointer is DEVICE memory on the current CUDA device, owned by
 *   the caller.  The library never allocates, frees or copies between host and
 *   device; it never synchronises the stream except in tgvkv_status.
 * - bf16 tensors are passed as raw 16-bit patterns (uint16_t).
 * - Every call is asynchronous on `stream` (a cudaStream_t passed as void*;
 *   NULL = the legacy default stream).
 * - Arguments are validated on the host before any launch; a bad argument
 *   returns TGVKV_ERR_INVALID_ARG / TGVKV_ERR_UNSUPPORTED and launches nothing.
 *   Data-dependent faults found on the device (a query position out of range,
 *   a modality mask that disagrees with N_v, a budget or index out of range,
 *   an on-chip wait that gave up) never trap: the kernel skips the bad access
 *   and sets a bit in the status word inside `workspace`, read back with
 *   tgvkv_status.
 * - The message of the last host-side error of the calling thread is returned
 *   by tgvkv_last_error.
 * - Pointers to bf16 tensors, `workspace`, and the outputs k_out/v_out must be
 *   16-byte aligned.
 *
 * Budget basis (desc->budget_basis).
 * - TGVKV_BASIS_VISION (the default): the ratio r is the fraction of VISION KV
 *   kept over all layers (the vision-only eviction setting of Appendix B.3,
 *   where the TPR policy keeps every text KV): B_V = floor(r * N_v * L + 1/2)
 *   vision rows per head are shared out over the layers.  Every KV head of
 *   layer l keeps the N_t text rows and b_l vision rows, so the compacted
 *   cache holds H_kv * (L * N_t + B_V) rows.
 * - TGVKV_BASIS_ALL: r is the fraction of ALL KV kept (the main-text setting,
 *   Section 4.3 / Table 4): B = floor(r * N * L + 1/2) rows per head are
 *   shared out (cap N per layer), and Eq. 10 applies per layer: b_l > N_t keeps
 *   every text row and the top (b_l - N_t) vision rows by the Eq. 8 score;
 *   b_l <= N_t keeps the top b_l text rows by the Eq. 9 score and no vision.
 * Sink tokens (desc->keep_first, desc->keep_last; Appendix A.2 keeps the first
 * 4 and the last token for every method): always kept, each taking one slot of
 * its own modality's part of the budget while slots remain.  Without sinks
 * the cache holds exactly H_kv * (L * N_t + B_V) (vision basis) or H_kv * B
 * (all-token basis) rows; sinks may add up to one row per sink per (l, g).
 * tgvkv_retained_rows gives the capacity, offsets[L*H_kv] the rows written.
 *
 * Budget statistic (desc->budget_stat; the layer-budget policies of Table 1a
 * and Eq. 5 with x in {VV, TV, TT}): TV (the method, default), TT (the
 * text-text mass of the query rows; tgvkv_evict runs the text-key pass and
 * returns that statistic in tvb_stat), or UNIFORM (no statistic).  VV, the
 * vision-vision mass, needs the vision tokens' queries: call tgvkv_score with
 * those queries as the rows (text_pos = the vision positions); its tvb_stat is
 * then the VV statistic, to split with tgvkv_budget.  The TT statistic of a
 * layer is also G * sum_{g,t} text_scores[l][g][t] (tgvkv_text_scores).
 *
 * Head-adaptive budgets (desc->head_budgets = 1; an extension -- the paper
 * budgets per layer only, Section 3.2): the statistic of (l, g) is the TV mass
 * of its G query heads (tvb_stat[l*H_kv+g]), H_kv * B rows are split over the
 * L * H_kv heads by the same rule (cap N_v, or N under the all-token basis),
 * and set (l, g) keeps budgets[l*H_kv+g].  With TGVKV_STAT_UNIFORM the split
 * is uniform over heads; TGVKV_STAT_TT is not supported.  At most 1024 heads.
 *
 * Text weights (desc->weight_mode): TGVKV_WEIGHTS_GIVEN uses the caller's w~
 * (Eq. 8); TGVKV_WEIGHTS_EQ7 makes tgvkv_evict derive w~ from the text-text
 * attention by Eq. 7 (tgvkv_text_scores) and ignore `w`.
 */
#ifndef TGVKV_H
#define TGVKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes ---------------------------------------------------- */
#define TGVKV_OK              0
#define TGVKV_ERR_INVALID_ARG 1   /* null / misaligned pointer, bad size or ratio */
#define TGVKV_ERR_UNSUPPORTED 2   /* a shape this build does not handle (e.g. d) */
#define TGVKV_ERR_CUDA        3   /* a CUDA runtime call failed (see last_error) */
#define TGVKV_ERR_DEVICE      4   /* tgvkv_status found device status bits set */

/* ---- device status bits (tgvkv_status) ------------------------------- */
#define TGVKV_STATUS_TEXT_POS     0x01u /* text_pos not strictly ascending or outside [0, N) */
#define TGVKV_STATUS_VISION_COUNT 0x02u /* modality marks a vision count other than N_v */
#define TGVKV_STATUS_BUDGET       0x04u /* a layer budget outside [0, N_v] reached select */
#define TGVKV_STATUS_INDEX        0x08u /* compact: an index outside [0, N), decreasing offsets, or a CSR larger than the output; decode: a CSR outside its rows */
#define TGVKV_STATUS_COUNT        0x10u /* a retained set did not hold N_t + b_l rows */
#define TGVKV_STATUS_TIMEOUT      0x20u /* a bounded on-chip wait gave up */
#define TGVKV_STATUS_WEIGHT       0x40u /* a text weight is negative or not finite */

/* ---- modes ------------------------------------------------------------ */
#define TGVKV_BASIS_VISION  0   /* r counts vision KV; all text KV kept (default) */
#define TGVKV_BASIS_ALL     1   /* r counts all KV; both cases of Eq. 10 */
#define TGVKV_WEIGHTS_GIVEN 0   /* the caller's normalised text weights w~ (default) */
#define TGVKV_WEIGHTS_EQ7   1   /* tgvkv_evict derives w~ by Eq. 7 */
#define TGVKV_STAT_TV       0   /* budgets follow the text-vision mass (Eq. 5, x = TV; default) */
#define TGVKV_STAT_TT       1   /* ... the text-text mass (x = TT, Table 1a) */
#define TGVKV_STAT_UNIFORM  2   /* ... no statistic: the uniform split of Table 1a */

/* ---- problem description --------------------------------------------- */
typedef struct tgvkv_desc {
    int32_t L;              /* decoder layers */
    int32_t H_q;            /* query heads per layer */
    int32_t H_kv;           /* KV heads per layer; H_q % H_kv == 0, G = H_q / H_kv */
    int32_t d;              /* head dimension: 64 or 128 */
    int32_t N;              /* cached tokens per layer and head (text + vision) */
    int32_t N_v;            /* vision tokens among them (N_t = N - N_v text tokens) */
    int32_t n_win;          /* text query rows (positions in text_pos) */
    float   softmax_scale;  /* logits = softmax_scale * <q, k>; <= 0 means 1/sqrt(d) */
    int64_t w_layer_stride; /* floats between the weight rows of two layers; 0 = one
                               row shared by every layer */
    int32_t budget_basis;   /* TGVKV_BASIS_VISION (0) or TGVKV_BASIS_ALL */
    int32_t weight_mode;    /* TGVKV_WEIGHTS_GIVEN (0) or TGVKV_WEIGHTS_EQ7 (tgvkv_evict) */
    int32_t keep_first;     /* sinks: the first keep_first positions are always kept */
    int32_t keep_last;      /* ... and the last keep_last positions */
    int32_t budget_stat;    /* TGVKV_STAT_TV (0), TGVKV_STAT_TT or TGVKV_STAT_UNIFORM */
    int32_t head_budgets;   /* 1: one budget per (layer, KV head); tvb_stat and budgets
                               then hold L * H_kv entries (head-major within a layer) */
} tgvkv_desc;

/* Size limits.  Every call checks the descriptor first and returns
 * TGVKV_ERR_UNSUPPORTED, launching nothing, when a limit is exceeded:
 *   N <= 32768 key positions per KV head (the score kernel holds a head's
 *     per-tile vision tables in shared memory);
 *   L <= 1024 layers;
 *   G * n_win <= 32768 query rows per KV head;
 *   L * H_kv <= 65535 KV heads in all (with head_budgets: <= 1024);
 *   d = 64 or 128.
 * TGVKV_ERR_INVALID_ARG covers the rest: non-positive L, H_q, H_kv or N,
 * N_v outside [0, N], n_win < 0, H_q not a multiple of H_kv, an unknown mode. */

/* Bytes of device workspace the calls below need for this problem (0 when the
 * descriptor is rejected). */
size_t tgvkv_workspace_size(const tgvkv_desc* desc);

/* B_V = floor(ratio * N_v * L + 1/2): vision rows kept per KV head over all
 * layers (Eq. 5 splits it).  Returns -1 if desc or ratio (not in [0,1]) is bad. */
int64_t tgvkv_vision_budget_total(const tgvkv_desc* desc, double ratio);

/* B of the descriptor's budget basis: B_V (vision basis) or
 * floor(ratio * N * L + 1/2) rows of any modality (all-token basis).
 * Returns -1 on bad arguments. */
int64_t tgvkv_budget_total(const tgvkv_desc* desc, double ratio);

/* Capacity of the compacted cache that idx, k_out and v_out must have:
 * H_kv * (L * N_t + B_V) (vision basis) or H_kv * B (all-token basis), plus
 * H_kv * L * (keep_first + keep_last) when there are sinks.  Returns -1 on bad
 * arguments. */
int64_t tgvkv_retained_rows(const tgvkv_desc* desc, double ratio);

/* TWR scores and the TVB statistic (Eq. 2, 5, 6, 8).
 *
 * For every layer l and query head h (KV head g = h / G), every query row i at
 * sequence position text_pos[i] attends causally to the keys 0..text_pos[i]
 * with A = softmax(softmax_scale * q k^T) over ALL of those keys (Eq. 2); the
 * text-vision attention is the slice of A on vision keys (Eq. 6).
 *   scores[l][g][v] = (1/G) sum_{h in g} sum_i w[l][i] * A_{l,h}[i, v]   (Eq. 8)
 *   tvb_stat[l]     = sum_h sum_i sum_v A_{l,h}[i, v]       (Eq. 5 numerator)
 * where v = 0..N_v-1 runs over the vision keys in position order.
 *
 * q_text:   bf16 [L][H_q][n_win][d]
 * k:        bf16 [L][H_kv][N][d]          (the key cache)
 * modality: uint8 [N], 1 = vision token, 0 = text token (same for all layers)
 * text_pos: int32 [n_win], strictly ascending positions in [0, N)
 * w:        fp32 text weights w~ >= 0, row l at w + l * w_layer_stride, n_win floats
 * scores:   fp32 [L][H_kv][N_v]  (output)
 * tvb_stat: fp32 [L]             (output; [L][H_kv], the per-head masses, with
 *           head budgets)
 * Arithmetic: bf16 products, fp32 accumulation and fp32 softmax. */
int tgvkv_score(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                const uint8_t* modality, const int32_t* text_pos, const float* w,
                float* scores, float* tvb_stat, void* workspace, void* stream);

/* Text scores (Eq. 9) and derived text weights (Eq. 7).
 *
 * From the same causal attention rows as tgvkv_score (Eq. 2), sliced on the
 * text keys (the text-text block A^(TT)):
 *   text_scores[l][g][t] = (1/G) sum_{h in g} sum_i A_{l,h}[i, t]          (Eq. 9)
 *   w_{l,j} = (1/H_q) sum_h sum_{i >= j} A_{l,h}[i, text_pos[j]] / (n_win - j)   (Eq. 7)
 *   weights[l][j] = w_{l,j} / sum_j' w_{l,j'}      (the normalised w~)
 * t runs over the text keys in position order; the rows i are the query rows
 * (rows before key t see it as 0 through the causal mask).  Every query row
 * must sit on a text token (else TGVKV_STATUS_TEXT_POS and a zero weight).
 * text_scores: fp32 [L][H_kv][N_t] (output); weights: fp32 [L][n_win]
 * (output; pass it to tgvkv_score as w with w_layer_stride = n_win).
 * Other arguments as in tgvkv_score. */
int tgvkv_text_scores(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                      const uint8_t* modality, const int32_t* text_pos,
                      float* text_scores, float* weights, void* workspace, void* stream);

/* TVB layer budgets (Eq. 5, x = TV).  Splits B_V over the layers in proportion
 * to tvb_stat: b_l = floor(B_V * S_l / sum S) plus one leftover unit each for
 * the largest fractional parts (ties: lower layer); a layer above N_v is capped
 * at N_v and the rest re-split over the other layers; all-zero statistics give a
 * uniform split.  The quotients are computed in double on the device.  Under
 * the all-token basis the same rule splits B with cap N.  With
 * TGVKV_STAT_UNIFORM the statistic is not read (tvb_stat may be NULL).
 * tvb_stat: fp32 [L]; budgets: int32 [L] (output, rows per KV head: vision rows
 * under the vision basis, rows of any modality under the all-token basis). */
int tgvkv_budget(const tgvkv_desc* desc, const float* tvb_stat, double ratio,
                 int32_t* budgets, void* workspace, void* stream);

/* TPR retention (Eq. 10, case b_l > N_t with the vision budget b_l).
 * For every (l, g): every text position plus the budgets[l] vision positions
 * with the largest scores[l][g][.] (ties: lower position), in ascending
 * position order.  The sets are stored as CSR over (l, g) in row-major order:
 * set (l, g) is idx[offsets[l*H_kv+g] .. offsets[l*H_kv+g+1]).
 * offsets: int64 [L*H_kv + 1] (output); idx: int32 positions (output, capacity
 * tgvkv_retained_rows). */
int tgvkv_select(const tgvkv_desc* desc, const float* scores, const int32_t* budgets,
                 const uint8_t* modality, int64_t* offsets, int32_t* idx,
                 void* workspace, void* stream);

/* TPR retention with every option of the descriptor (Eq. 10, both cases,
 * sinks).  As tgvkv_select, plus text_scores: fp32 [L][H_kv][N_t] from
 * tgvkv_text_scores, read for the layers with b_l <= N_t under the all-token
 * basis (may be NULL under the vision basis).  tgvkv_select is this call with
 * text_scores = NULL; it rejects the all-token basis. */
int tgvkv_select_tpr(const tgvkv_desc* desc, const float* scores, const float* text_scores,
                     const int32_t* budgets, const uint8_t* modality, int64_t* offsets,
                     int32_t* idx, void* workspace, void* stream);

/* Compaction: row r of set (l, g) of the CSR becomes
 *   k_out[r] = k[l][g][idx[r]],  v_out[r] = v[l][g][idx[r]]
 * as bit copies.  k, v: bf16 [L][H_kv][N][d]; k_out, v_out: bf16
 * [capacity_rows][d] (output; rows 0 .. offsets[L*H_kv] are written, and
 * tgvkv_retained_rows rows always suffice for sets tgvkv_select made).
 * capacity_rows: rows the caller allocated in each of k_out and v_out (>= 0).
 * A CSR whose total offsets[L*H_kv] is negative or above capacity_rows sets
 * TGVKV_STATUS_INDEX and only rows below capacity_rows are written; an
 * idx entry outside [0, N) sets the same bit and its row is skipped. */
int tgvkv_compact(const tgvkv_desc* desc, const uint16_t* k, const uint16_t* v,
                  const int64_t* offsets, const int32_t* idx,
                  uint16_t* k_out, uint16_t* v_out, int64_t capacity_rows,
                  void* workspace, void* stream);

/* TPR retention and compaction in one pass (Eq. 10, then the gather): the
 * tail of tgvkv_evict for scores and budgets the caller already holds.  The
 * sets are those tgvkv_select_tpr makes (every option of the descriptor) and
 * their rows those tgvkv_compact copies: offsets, idx, k_out and v_out as in
 * those two calls.  scores, text_scores, budgets, modality: as in
 * tgvkv_select_tpr; k, v: as in tgvkv_compact.
 * capacity_rows: rows the caller allocated in each of idx, k_out and v_out
 * (>= 0; tgvkv_retained_rows always suffices for budgets tgvkv_budget split
 * from a ratio).  A set that would end past capacity_rows sets
 * TGVKV_STATUS_INDEX and none of its indices or rows is written (offsets are
 * written in full); a budget outside [0, cap] sets TGVKV_STATUS_BUDGET and is
 * clamped.  One kernel for most shapes, or select then compact for sets too
 * large for shared memory (tgvkv_select_compact_launches). */
int tgvkv_select_compact(const tgvkv_desc* desc, const float* scores, const float* text_scores,
                         const int32_t* budgets, const uint8_t* modality, const uint16_t* k,
                         const uint16_t* v, int64_t* offsets, int32_t* idx, uint16_t* k_out,
                         uint16_t* v_out, int64_t capacity_rows, void* workspace, void* stream);

/* Kernel launches one tgvkv_select_compact call makes for desc (1 or 2; -1 on
 * an invalid descriptor). */
int tgvkv_select_compact_launches(const tgvkv_desc* desc);

/* score -> budget -> select -> compact in one stream-ordered call with no host
 * synchronisation.  Arguments as in the four calls above.  With Eq. 7 weights
 * or the all-token basis it first runs tgvkv_text_scores into the workspace
 * (`w` is then ignored under TGVKV_WEIGHTS_EQ7). */
int tgvkv_evict(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                const float* w, double ratio,
                float* scores, float* tvb_stat, int32_t* budgets,
                int64_t* offsets, int32_t* idx, uint16_t* k_out, uint16_t* v_out,
                void* workspace, void* stream);

/* Causal prefill attention over every token, which also keeps what the
 * eviction step needs from the rows at its query positions (the prefill phase
 * of Section 3.1: Eq. 2 over all N rows; Eq. 5 / Eq. 6 read the same rows).
 *
 * For every layer l, query head h (KV head g = h / G) and token i:
 *   o[l][h][i][:] = sum_{j <= i} softmax_j(softmax_scale <q[l][h][i], k[l][g][j]>) v[l][g][j][:]
 * and for every query row r of the eviction step (position p = text_pos[r]):
 *   q_text[l][h][r][:]  = q[l][h][p][:]                      (bit copy)
 *   row_stats[l][h][r]  = (m, Z, V):  Z = sum_{j <= p} 2^(x_pj log2(e) - m),
 *                         V = the same sum over the vision keys j,
 *                         x_pj = softmax_scale <q[l][h][p], k[l][g][j]>,
 *                         m = a reference value at most 8 below the row's
 *                         largest x_pj log2(e) and not above it.
 * q: bf16 [L][H_q][N][d]; k, v: bf16 [L][H_kv][N][d]; modality: uint8 [N];
 * text_pos: int32 [n_win] strictly ascending (may be NULL when n_win = 0);
 * o: bf16 [L][H_q][N][d] (output); q_text: bf16 [L][H_q][n_win][d] (output);
 * row_stats: fp32 [L][H_q][n_win][3] (output).  q, k, v, o and q_text must be
 * 16-byte aligned.  bf16 products with fp32 accumulation and softmax; the
 * attention weights enter the value product rounded to bf16, and o is rounded
 * to bf16.  q_text and row_stats are the inputs tgvkv_evict_with_stats takes.
 * Device-side checks: text_pos (TGVKV_STATUS_TEXT_POS), bounded waits
 * (TGVKV_STATUS_TIMEOUT). */
int tgvkv_prefill(const tgvkv_desc* desc, const uint16_t* q, const uint16_t* k,
                  const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                  uint16_t* o, uint16_t* q_text, float* row_stats, void* workspace,
                  void* stream);

/* tgvkv_evict with the query rows' statistics given: row_stats as tgvkv_prefill
 * writes them (fp32 [L][H_q][n_win][3]).  The score passes then read each
 * row's (m, Z, vision mass) instead of streaming its keys a first time; all
 * other arguments and every result are those of tgvkv_evict.  Under TT
 * budgeting the text-key pass keeps its own row statistics (its statistic is
 * each row's text mass, which row_stats does not hold); the vision pass reads
 * the given ones. */
int tgvkv_evict_with_stats(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                           const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                           const float* w, double ratio, const float* row_stats,
                           float* scores, float* tvb_stat, int32_t* budgets,
                           int64_t* offsets, int32_t* idx, uint16_t* k_out, uint16_t* v_out,
                           void* workspace, void* stream);

/* Number of CUDA kernels one tgvkv_evict call launches for this problem
 * (introspection for callers that budget launches, e.g. inside a captured
 * graph; the paper has no counterpart): normally 2 (scores with the layer
 * budgets, then select + gather fused), 3 when the fused kernel's
 * shared-memory table does not fit (select and compact separately); 2 more
 * (the text-key score pass and the Eq. 7 weights) with Eq. 7 weights or the
 * all-token basis.  A problem
 * with no query rows zero-fills the scores with memsets and launches the
 * budget kernel in place of the score kernel.  Returns -1 on bad arguments. */
int tgvkv_evict_launches(const tgvkv_desc* desc);

/* Decode over the compacted cache (the consumer of the eviction step; the
 * decode phase of Section 3.1).  For one new token per layer, query head h of
 * layer l attends to the rows of set (l, g = h / G) of a CSR cache:
 *   out[l][h][:] = sum_r softmax_r(softmax_scale * <q[l][h], k_rows[r]>) v_rows[r]
 * over r in [offsets[l*H_kv+g], offsets[l*H_kv+g+1]); an empty set gives 0.
 * q: bf16 [L][H_q][d], 16-byte aligned; k_rows, v_rows: bf16 [rows][d], 16-byte
 * aligned (k_out / v_out of tgvkv_evict, or the full cache [L][H_kv][N][d]
 * with offsets[i] = i * N), each holding at least capacity_rows rows;
 * offsets: int64 [L*H_kv + 1], nondecreasing; out: fp32 [L][H_q][d] (output),
 * 8-byte aligned.  bf16 products, fp32 accumulation and softmax; the softmax
 * weights enter the value sum as bf16(P) + bf16(P - bf16(P)) (about 16 bits).
 * Rows at or above capacity_rows (and above 2^31 - 1) are never read: a set
 * that reaches them, or a decreasing or negative offset, sets
 * TGVKV_STATUS_INDEX (results then undefined).  capacity_rows < 0 is
 * rejected.  The rows of other sets
 * next to a set's own may be read and are masked: they must be finite.
 * Two kernels: the row streams, then (launched as a programmatic dependent)
 * the merge of the sets they split; the workspace holds the streams' partial
 * results (tgvkv_workspace_size covers them). */
int tgvkv_decode(const tgvkv_desc* desc, const uint16_t* q, const uint16_t* k_rows,
                 const uint16_t* v_rows, int64_t capacity_rows, const int64_t* offsets,
                 float* out, void* workspace, void* stream);

/* Kernels one tgvkv_decode call launches (2).  -1 on bad arguments. */
int tgvkv_decode_launches(const tgvkv_desc* desc);

/* Zero `workspace` (asynchronously on `stream`).  Needed once after the
 * workspace is allocated: the calls leave their completion counters at zero
 * for the next call.  Zero it again after a call whose tgvkv_status reported
 * TGVKV_STATUS_TIMEOUT, and never share one workspace between calls that may
 * overlap on the GPU. */
int tgvkv_workspace_init(const tgvkv_desc* desc, void* workspace, void* stream);

/* Synchronise `stream`, then read and clear the device status word kept in
 * `workspace`.  Returns the TGVKV_STATUS_* bits (0 = clean) or a negative
 * value if the synchronisation itself failed. */
int tgvkv_status(void* workspace, void* stream);

/* Self-test of the failure detection (no counterpart in the paper).  Launches
 * one CTA that waits, with the same bounded wait every kernel of the library
 * uses, on an mbarrier that nothing arrives at.  The wait gives up after its
 * limit (2e9 SM cycles, about 1 s) and the kernel sets TGVKV_STATUS_TIMEOUT in
 * the status word of `workspace`, which tgvkv_status then returns; nothing
 * faults and the context stays usable.  Returns TGVKV_OK once launched. */
int tgvkv_check_wait_timeout(void* workspace, void* stream);

/* Message of the last error returned on the calling thread ("" if none). */
const char* tgvkv_last_error(void);

/* tgvkv_score without a caller workspace (the paper has no counterpart; this
 * is a deployment variant of tgvkv_score).
 *
 * For callers that are handed only input and output buffers and cannot
 * allocate device memory themselves: for example a plugin inside an inference
 * runtime that owns all device memory and passes its operators no workspace,
 * or a latency-critical path where cudaMalloc's implicit synchronisation is
 * not allowed.  The scratch this call needs (completion counters, per-tile
 * partial scores and TV masses) lives in a fixed array of
 * TGVKV_NOALLOC_SCRATCH_BYTES inside the library; every GPU that loads the
 * library holds that array until the process exits.  Nothing is allocated.
 *
 * Same arguments and results as tgvkv_score, minus the workspace.
 * - A problem whose scratch (the part of the tgvkv_workspace_size workspace
 *   that tgvkv_score uses: all of it but the decode partials at its end)
 *   exceeds TGVKV_NOALLOC_SCRATCH_BYTES is rejected with
 *   TGVKV_ERR_UNSUPPORTED before any launch.
 * - Every call looks up the array's device address in the current device's
 *   context (so a context created after cudaDeviceReset uses its own array);
 *   the first call on a device may load the library's device code, so make it
 *   before any stream capture.
 * - All calls share the one array.  Each call clears the parts that must start
 *   at zero; calls whose work overlaps on the GPU (different streams, or
 *   different host threads, on one device) race on the array and must be
 *   serialised by the caller.
 * - The device status word is kept in the array: each call clears it before
 *   its launch, so after a call tgvkv_noalloc_status returns that call's
 *   TGVKV_STATUS_* bits (input faults that were skipped, and
 *   TGVKV_STATUS_TIMEOUT when a bounded wait gave up and the scores are
 *   unfinished).  Read it before the next call clears it. */
#define TGVKV_NOALLOC_SCRATCH_BYTES (8u << 20)
int tgvkv_score_noalloc(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                        const uint8_t* modality, const int32_t* text_pos, const float* w,
                        float* scores, float* tvb_stat, void* stream);

/* Synchronise `stream`, then read and clear the status word of
 * tgvkv_score_noalloc's fixed array on the current device (the counterpart of
 * tgvkv_status for that call).  Returns the TGVKV_STATUS_* bits (0 = clean)
 * or a negative error code.  Allocates nothing. */
int tgvkv_noalloc_status(void* stream);

#ifdef __cplusplus
}
#endif
#endif /* TGVKV_H */
