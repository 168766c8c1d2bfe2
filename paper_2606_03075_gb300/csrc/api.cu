// C ABI of the TGV-KV eviction step: argument checks on the host, workspace
// layout, and the stream-ordered launches of the four kernels.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>

#include "common.cuh"
#include "launch.h"
#include "tgvkv.h"

namespace tgvkv {
namespace {

thread_local char g_last_error[512] = "";

int fail(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
    return code;
}

int ok() {
    g_last_error[0] = '\0';
    return TGVKV_OK;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(TGVKV_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

size_t round_up(size_t x) { return (x + 255) & ~size_t(255); }

// tgvkv_evict needs the Eq. 9 text scores: for Eq. 7 weights, or for case
// b_l <= N_t of Eq. 10 under the all-token basis.
bool needs_text_pass(const Problem& p) {
    return p.weights_eq7 || p.basis == TGVKV_BASIS_ALL || p.budget_stat == TGVKV_STAT_TT;
}

WsLayout layout_of(const Problem& p) {
    WsLayout w;
    size_t o = 0;
    w.status = o;      o += round_up(sizeof(uint32_t));
    w.tickets = o;     o += round_up(sizeof(uint32_t) * ticket_words(p));
    w.stat_part = o;   o += round_up(sizeof(float) * (size_t)p.L * p.H_kv * (p.T > 0 ? p.T : 1));
    w.stat_head = o;   o += round_up(sizeof(float) * (size_t)p.L * p.H_kv);
    w.score_part = o;
    const size_t keyset = (size_t)(p.N_v > p.N_t ? p.N_v : p.N_t);
    if (p.T > 1) o += round_up(sizeof(float) * (size_t)p.L * p.H_kv * p.T * keyset);
    w.stat_text = o;   o += round_up(sizeof(float) * (size_t)p.L);
    w.text_scores = w.weights = w.row_stats = 0;
    if (needs_text_pass(p)) {
        w.text_scores = o; o += round_up(sizeof(float) * (size_t)p.L * p.H_kv * (p.N_t > 0 ? p.N_t : 1));
        w.weights = o;     o += round_up(sizeof(float) * (size_t)p.L * (p.n_win > 0 ? p.n_win : 1));
        w.row_stats = o;   o += round_up(3 * sizeof(float) * ((size_t)p.L * p.H_q * p.n_win + 1));
    }
    w.score_total = o;
    // decode only, after everything the score and eviction calls use
    w.decode_part = o;
    o += round_up(sizeof(float) * (size_t)decode_passes(p) * kDecMaxStreams * 2 *
                  decode_record_floats(p));
    w.total = o;
    return w;
}

// Validate a descriptor and build the kernels' view of it.
int make_problem(const tgvkv_desc* d, Problem* p) {
    if (!d) return fail(TGVKV_ERR_INVALID_ARG, "desc is NULL");
    if (d->L < 1 || d->H_q < 1 || d->H_kv < 1 || d->N < 1 || d->n_win < 0 || d->N_v < 0 ||
        d->N_v > d->N)
        return fail(TGVKV_ERR_INVALID_ARG,
                    "bad sizes: L=%d H_q=%d H_kv=%d N=%d N_v=%d n_win=%d", d->L, d->H_q, d->H_kv,
                    d->N, d->N_v, d->n_win);
    if (d->H_q % d->H_kv != 0)
        return fail(TGVKV_ERR_INVALID_ARG, "H_q=%d is not a multiple of H_kv=%d", d->H_q, d->H_kv);
    if (d->d != 64 && d->d != 128)
        return fail(TGVKV_ERR_UNSUPPORTED, "head dim %d unsupported (64 or 128)", d->d);
    if (d->N > kMaxN) return fail(TGVKV_ERR_UNSUPPORTED, "N=%d above %d", d->N, kMaxN);
    if (d->N_v > kMaxNv) return fail(TGVKV_ERR_UNSUPPORTED, "N_v=%d above %d", d->N_v, kMaxNv);
    if (d->L > kMaxL) return fail(TGVKV_ERR_UNSUPPORTED, "L=%d above %d", d->L, kMaxL);
    if (d->w_layer_stride < 0)
        return fail(TGVKV_ERR_INVALID_ARG, "w_layer_stride=%lld < 0", (long long)d->w_layer_stride);
    if (!(d->softmax_scale == d->softmax_scale) || isinf(d->softmax_scale))
        return fail(TGVKV_ERR_INVALID_ARG, "softmax_scale is not finite");
    const long long rows = (long long)(d->H_q / d->H_kv) * d->n_win;
    if (rows > 32768) return fail(TGVKV_ERR_UNSUPPORTED, "G * n_win = %lld above 32768", rows);
    if ((long long)d->L * d->H_kv > 65535)
        return fail(TGVKV_ERR_UNSUPPORTED, "L * H_kv above 65535");
    if ((long long)d->L * d->H_kv * d->N >= (1LL << 31) ||
        (long long)d->L * d->H_q * d->n_win >= (1LL << 31))
        return fail(TGVKV_ERR_UNSUPPORTED, "K or Q holds 2^31 rows or more");
    p->L = d->L;
    p->H_q = d->H_q;
    p->H_kv = d->H_kv;
    p->G = d->H_q / d->H_kv;
    p->d = d->d;
    p->N = d->N;
    p->N_v = d->N_v;
    p->N_t = d->N - d->N_v;
    p->n_win = d->n_win;
    p->R = (int)rows;
    p->T = (p->R + 127) / 128;
    const double scale = d->softmax_scale > 0.f ? (double)d->softmax_scale : 1.0 / sqrt((double)d->d);
    p->scale_log2 = (float)(scale * 1.4426950408889634);  // log2(e)
    p->w_stride = (long long)d->w_layer_stride;
    if (d->budget_basis != TGVKV_BASIS_VISION && d->budget_basis != TGVKV_BASIS_ALL)
        return fail(TGVKV_ERR_INVALID_ARG, "budget_basis=%d unknown", d->budget_basis);
    if (d->weight_mode != TGVKV_WEIGHTS_GIVEN && d->weight_mode != TGVKV_WEIGHTS_EQ7)
        return fail(TGVKV_ERR_INVALID_ARG, "weight_mode=%d unknown", d->weight_mode);
    if (d->keep_first < 0 || d->keep_last < 0)
        return fail(TGVKV_ERR_INVALID_ARG, "keep_first=%d / keep_last=%d < 0", d->keep_first,
                    d->keep_last);
    p->basis = d->budget_basis;
    p->weights_eq7 = d->weight_mode == TGVKV_WEIGHTS_EQ7;
    p->keep_first = d->keep_first < d->N ? d->keep_first : d->N;
    p->keep_last = d->keep_last < d->N ? d->keep_last : d->N;
    if (d->budget_stat != TGVKV_STAT_TV && d->budget_stat != TGVKV_STAT_TT &&
        d->budget_stat != TGVKV_STAT_UNIFORM)
        return fail(TGVKV_ERR_INVALID_ARG, "budget_stat=%d unknown", d->budget_stat);
    p->budget_stat = d->budget_stat;
    if (d->head_budgets != 0 && d->head_budgets != 1)
        return fail(TGVKV_ERR_INVALID_ARG, "head_budgets=%d is neither 0 nor 1", d->head_budgets);
    p->head_budgets = d->head_budgets;
    if (p->head_budgets && p->budget_stat == TGVKV_STAT_TT)
        return fail(TGVKV_ERR_UNSUPPORTED, "head budgets follow the TV mass or are uniform");
    if (p->head_budgets && (long long)p->L * p->H_kv > kMaxL)
        return fail(TGVKV_ERR_UNSUPPORTED, "head budgets for L * H_kv = %d heads above %d",
                    p->L * p->H_kv, kMaxL);
    p->keys_text = 0;
    p->row_stats = nullptr;
    p->stats_given = 0;
    return TGVKV_OK;
}

int check_ratio(double ratio) {
    if (!(ratio >= 0.0 && ratio <= 1.0))
        return fail(TGVKV_ERR_INVALID_ARG, "ratio %g outside [0, 1]", ratio);
    return TGVKV_OK;
}

long long vision_budget_total(const Problem& p, double ratio) {
    return (long long)floor(ratio * (double)((long long)p.N_v * p.L) + 0.5);
}

// B: rows per head over all layers that the budget split shares out --
// vision rows (vision basis) or rows of any modality (all-token basis).
long long budget_total(const Problem& p, double ratio) {
    if (p.basis == TGVKV_BASIS_ALL) return (long long)floor(ratio * (double)((long long)p.N * p.L) + 0.5);
    return vision_budget_total(p, ratio);
}

// Units the budget split shares out: per head, H_kv times the rows per head.
long long split_total(const Problem& p, double ratio) {
    return p.head_budgets ? (long long)p.H_kv * budget_total(p, ratio) : budget_total(p, ratio);
}

// Sink positions (at most N).
int n_sinks(const Problem& p) {
    const int both = p.keep_first + p.keep_last;
    return both < p.N ? both : p.N;
}

// Capacity of the compacted cache.  Exact without sinks: H_kv * (L * N_t + B_V)
// (vision basis) or H_kv * B (all-token basis).  A sink can add one row above a
// layer's budget, so sinks add at most H_kv * L * (keep_first + keep_last).
long long retained_rows(const Problem& p, double ratio) {
    const long long base = p.basis == TGVKV_BASIS_ALL
                               ? budget_total(p, ratio)
                               : (long long)p.L * p.N_t + budget_total(p, ratio);
    return (long long)p.H_kv * (base + (long long)p.L * n_sinks(p));
}

#define REQUIRE_PTR(ptr, name, need16)                                                   \
    do {                                                                                 \
        if (!(ptr)) return fail(TGVKV_ERR_INVALID_ARG, "%s is NULL", name);              \
        if ((need16) && !aligned16(ptr))                                                 \
            return fail(TGVKV_ERR_INVALID_ARG, "%s is not 16-byte aligned", name);       \
    } while (0)

uint32_t* status_of(void* ws, const WsLayout& lay) {
    return reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + lay.status);
}

int do_score(const Problem& p, const uint16_t* q, const uint16_t* k, const uint8_t* modality,
             const int32_t* text_pos, const float* w, float* scores, float* tvb_stat, void* ws,
             cudaStream_t st) {
    const WsLayout lay = layout_of(p);
    cudaError_t e = launch_score(p, q, k, modality, text_pos, w, scores, tvb_stat,
                                 static_cast<char*>(ws), lay, -1, nullptr, st);
    return e == cudaSuccess ? TGVKV_OK : cuda_fail(e, "score launch");
}

// The problem of the text-key pass (Eq. 9): the score kernel with the key set
// and its size swapped to the text keys.
Problem text_problem(const Problem& p) {
    Problem t = p;
    t.keys_text = 1;
    t.N_v = p.N_t;
    t.N_t = p.N_v;
    return t;
}

// Eq. 9 text scores and Eq. 7 weights: the text-key score pass, then the
// per-layer weights.  stat_scratch takes the pass's (unused) statistic.
int do_text_scores(const Problem& p, const uint16_t* q, const uint16_t* k, const uint8_t* modality,
                   const int32_t* text_pos, float* text_scores, float* weights, float* stat_out,
                   void* ws, cudaStream_t st, long long budget_total = -1, int32_t* budgets = nullptr,
                   float* row_stats = nullptr, bool stats_given = false) {
    const WsLayout lay = layout_of(p);
    Problem tp = text_problem(p);
    tp.row_stats = row_stats;
    tp.stats_given = stats_given ? 1 : 0;
    cudaError_t e = launch_score(tp, q, k, modality, text_pos, nullptr, text_scores, stat_out,
                                 static_cast<char*>(ws), lay, budget_total, budgets, st);
    if (e != cudaSuccess) return cuda_fail(e, "text-key score launch");
    if (weights) {
        e = launch_eq7_weights(p, text_scores, modality, text_pos, weights, status_of(ws, lay), st);
        if (e != cudaSuccess) return cuda_fail(e, "Eq. 7 weights launch");
    }
    return TGVKV_OK;
}

int check_score_args(const Problem& p, const uint16_t* q, const uint16_t* k,
                     const uint8_t* modality, const int32_t* text_pos, const float* w,
                     const float* scores, const float* tvb_stat, const void* ws,
                     bool need_w = true) {
    if (p.n_win > 0) {
        REQUIRE_PTR(q, "q_text", true);
        REQUIRE_PTR(text_pos, "text_pos", false);
        if (need_w) REQUIRE_PTR(w, "w", false);
    }
    REQUIRE_PTR(k, "k", true);
    REQUIRE_PTR(modality, "modality", false);
    if (p.N_v > 0) REQUIRE_PTR(scores, "scores", false);
    REQUIRE_PTR(tvb_stat, "tvb_stat", false);
    REQUIRE_PTR(ws, "workspace", true);
    return TGVKV_OK;
}

// tgvkv_evict, with the query rows' (m, Z, vision mass) computed by the score
// passes, or given by the caller (stats_given).
int evict_impl(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
               const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
               const float* w, double ratio, bool stats_given, const float* given_stats, float* scores,
               float* tvb_stat, int32_t* budgets, int64_t* offsets, int32_t* idx, uint16_t* k_out,
               uint16_t* v_out, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if ((rc = check_ratio(ratio))) return rc;
    if (stats_given && p.n_win > 0) REQUIRE_PTR(given_stats, "row_stats", false);
    // with no query rows (n_win = 0) no score pass runs and nothing is read
    float* stats = stats_given && p.n_win > 0 ? const_cast<float*>(given_stats) : nullptr;
    rc = check_score_args(p, q_text, k, modality, text_pos, w, scores, tvb_stat, workspace,
                          !p.weights_eq7);
    if (rc) return rc;
    REQUIRE_PTR(v, "v", true);
    REQUIRE_PTR(budgets, "budgets", false);
    REQUIRE_PTR(offsets, "offsets", false);
    REQUIRE_PTR(idx, "idx", false);
    REQUIRE_PTR(k_out, "k_out", true);
    REQUIRE_PTR(v_out, "v_out", true);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const WsLayout lay = layout_of(p);
    uint32_t* status = status_of(workspace, lay);
    char* wsb = static_cast<char*>(workspace);
    float* text_scores = nullptr;
    if (needs_text_pass(p)) {
        // Eq. 9 text scores (and Eq. 7 weights) into the workspace first
        text_scores = reinterpret_cast<float*>(wsb + lay.text_scores);
        float* wts = p.weights_eq7 ? reinterpret_cast<float*>(wsb + lay.weights) : nullptr;
        // with TT budgeting the text pass's statistic (the text-text mass) is the one
        // split, by that pass's last CTA
        const bool tt = p.budget_stat == TGVKV_STAT_TT;
        // the text-key pass computes the rows' (m, Z, vision mass) into the
        // workspace, or reads the given ones -- except under TT budgeting, whose
        // statistic is each row's text mass, which the given statistics do not
        // hold: then the text-key pass keeps its own row statistics
        const bool text_reads = stats != nullptr && !tt;
        rc = do_text_scores(p, q_text, k, modality, text_pos, text_scores, p.n_win > 0 ? wts : nullptr,
                            tt ? tvb_stat : reinterpret_cast<float*>(wsb + lay.stat_text), workspace, st,
                            tt ? split_total(p, ratio) : -1, tt ? budgets : nullptr,
                            text_reads ? stats : reinterpret_cast<float*>(wsb + lay.row_stats),
                            text_reads);
        if (rc) return rc;
    }
    Problem ps = p;
    if (stats || needs_text_pass(p)) {
        // the vision pass takes the rows' (m, Z, vision mass) from the caller or
        // the text-key pass instead of a pass A of its own
        ps.row_stats = stats ? stats : reinterpret_cast<float*>(wsb + lay.row_stats);
        ps.stats_given = 1;
    }
    const float* w_used = w;
    if (p.weights_eq7) {
        w_used = reinterpret_cast<const float*>(wsb + lay.weights);
        ps.w_stride = p.n_win;
    }
    // the score kernel's last CTA also derives the layer budgets (TV or uniform;
    // with TT budgeting the text pass did, and the TV statistic goes to scratch)
    const bool tt = p.budget_stat == TGVKV_STAT_TT;
    cudaError_t e = launch_score(ps, q_text, k, modality, text_pos, w_used, scores,
                                 tt ? reinterpret_cast<float*>(wsb + lay.stat_text) : tvb_stat, wsb,
                                 lay, split_total(p, ratio), tt ? nullptr : budgets, st);
    if (e != cudaSuccess) return cuda_fail(e, "score launch");
    if (score_launches(p) == 0) {   // no score kernel ran: split the (zero) statistic here
        e = launch_budget(p, tvb_stat, split_total(p, ratio), budgets, status, st);
        if (e != cudaSuccess) return cuda_fail(e, "budget launch");
    }
    e = launch_select_compact(p, scores, text_scores, budgets, modality, offsets, idx, k, v, k_out,
                              v_out, retained_rows(p, ratio), status, st);
    if (e != cudaSuccess) return cuda_fail(e, "select/compact launch");
    return ok();
}

}  // namespace
}  // namespace tgvkv

using namespace tgvkv;

extern "C" {

size_t tgvkv_workspace_size(const tgvkv_desc* desc) {
    Problem p{};
    if (make_problem(desc, &p) != TGVKV_OK) return 0;
    return layout_of(p).total;
}

int64_t tgvkv_vision_budget_total(const tgvkv_desc* desc, double ratio) {
    Problem p{};
    if (make_problem(desc, &p) != TGVKV_OK || check_ratio(ratio) != TGVKV_OK) return -1;
    return budget_total(p, ratio);
}

int64_t tgvkv_budget_total(const tgvkv_desc* desc, double ratio) {
    Problem p{};
    if (make_problem(desc, &p) != TGVKV_OK || check_ratio(ratio) != TGVKV_OK) return -1;
    return budget_total(p, ratio);
}

int64_t tgvkv_retained_rows(const tgvkv_desc* desc, double ratio) {
    Problem p{};
    if (make_problem(desc, &p) != TGVKV_OK || check_ratio(ratio) != TGVKV_OK) return -1;
    return retained_rows(p, ratio);
}

int tgvkv_score(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                const uint8_t* modality, const int32_t* text_pos, const float* w,
                float* scores, float* tvb_stat, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    rc = check_score_args(p, q_text, k, modality, text_pos, w, scores, tvb_stat, workspace);
    if (rc) return rc;
    rc = do_score(p, q_text, k, modality, text_pos, w, scores, tvb_stat, workspace,
                  static_cast<cudaStream_t>(stream));
    return rc ? rc : ok();
}

int tgvkv_text_scores(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                      const uint8_t* modality, const int32_t* text_pos, float* text_scores,
                      float* weights, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if (p.n_win > 0) {
        REQUIRE_PTR(q_text, "q_text", true);
        REQUIRE_PTR(text_pos, "text_pos", false);
        REQUIRE_PTR(weights, "weights", false);
    }
    REQUIRE_PTR(k, "k", true);
    REQUIRE_PTR(modality, "modality", false);
    if (p.N_t > 0) REQUIRE_PTR(text_scores, "text_scores", false);
    REQUIRE_PTR(workspace, "workspace", true);
    const WsLayout lay = layout_of(p);
    float* scratch = reinterpret_cast<float*>(static_cast<char*>(workspace) + lay.stat_text);
    rc = do_text_scores(p, q_text, k, modality, text_pos, text_scores, p.n_win > 0 ? weights : nullptr,
                        scratch, workspace, static_cast<cudaStream_t>(stream));
    return rc ? rc : ok();
}

int tgvkv_budget(const tgvkv_desc* desc, const float* tvb_stat, double ratio, int32_t* budgets,
                 void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if ((rc = check_ratio(ratio))) return rc;
    if (p.budget_stat != TGVKV_STAT_UNIFORM) REQUIRE_PTR(tvb_stat, "tvb_stat", false);
    REQUIRE_PTR(budgets, "budgets", false);
    REQUIRE_PTR(workspace, "workspace", true);
    const WsLayout lay = layout_of(p);
    cudaError_t e = launch_budget(p, tvb_stat, split_total(p, ratio), budgets,
                                  status_of(workspace, lay), static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "budget launch");
}

int tgvkv_select_tpr(const tgvkv_desc* desc, const float* scores, const float* text_scores,
                     const int32_t* budgets, const uint8_t* modality, int64_t* offsets,
                     int32_t* idx, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if (p.N_v > 0) REQUIRE_PTR(scores, "scores", false);
    if (p.basis == TGVKV_BASIS_ALL && p.N_t > 0) REQUIRE_PTR(text_scores, "text_scores", false);
    REQUIRE_PTR(budgets, "budgets", false);
    REQUIRE_PTR(modality, "modality", false);
    REQUIRE_PTR(offsets, "offsets", false);
    REQUIRE_PTR(idx, "idx", false);
    REQUIRE_PTR(workspace, "workspace", true);
    const WsLayout lay = layout_of(p);
    cudaError_t e = launch_select(p, scores, text_scores, budgets, modality, offsets, idx,
                                  status_of(workspace, lay), static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "select launch");
}

int tgvkv_select(const tgvkv_desc* desc, const float* scores, const int32_t* budgets,
                 const uint8_t* modality, int64_t* offsets, int32_t* idx, void* workspace,
                 void* stream) {
    if (desc && desc->budget_basis == TGVKV_BASIS_ALL)
        return fail(TGVKV_ERR_INVALID_ARG,
                    "the all-token basis needs the text scores: use tgvkv_select_tpr");
    return tgvkv_select_tpr(desc, scores, nullptr, budgets, modality, offsets, idx, workspace,
                            stream);
}

int tgvkv_compact(const tgvkv_desc* desc, const uint16_t* k, const uint16_t* v,
                  const int64_t* offsets, const int32_t* idx, uint16_t* k_out, uint16_t* v_out,
                  int64_t capacity_rows, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if (capacity_rows < 0) return fail(TGVKV_ERR_INVALID_ARG, "capacity_rows %lld < 0",
                                       (long long)capacity_rows);
    REQUIRE_PTR(k, "k", true);
    REQUIRE_PTR(v, "v", true);
    REQUIRE_PTR(offsets, "offsets", false);
    REQUIRE_PTR(idx, "idx", false);
    REQUIRE_PTR(k_out, "k_out", true);
    REQUIRE_PTR(v_out, "v_out", true);
    REQUIRE_PTR(workspace, "workspace", true);
    const WsLayout lay = layout_of(p);
    // every set holds at most N rows: no more can be asked of the kernel
    const long long cap = std::min((long long)capacity_rows, (long long)p.L * p.H_kv * p.N);
    cudaError_t e = launch_compact(p, k, v, offsets, idx, k_out, v_out, cap,
                                   status_of(workspace, lay), static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "compact launch");
}

int tgvkv_select_compact(const tgvkv_desc* desc, const float* scores, const float* text_scores,
                         const int32_t* budgets, const uint8_t* modality, const uint16_t* k,
                         const uint16_t* v, int64_t* offsets, int32_t* idx, uint16_t* k_out,
                         uint16_t* v_out, int64_t capacity_rows, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if (capacity_rows < 0) return fail(TGVKV_ERR_INVALID_ARG, "capacity_rows %lld < 0",
                                       (long long)capacity_rows);
    if (p.N_v > 0) REQUIRE_PTR(scores, "scores", false);
    if (p.basis == TGVKV_BASIS_ALL && p.N_t > 0) REQUIRE_PTR(text_scores, "text_scores", false);
    REQUIRE_PTR(budgets, "budgets", false);
    REQUIRE_PTR(modality, "modality", false);
    REQUIRE_PTR(k, "k", true);
    REQUIRE_PTR(v, "v", true);
    REQUIRE_PTR(offsets, "offsets", false);
    REQUIRE_PTR(idx, "idx", false);
    REQUIRE_PTR(k_out, "k_out", true);
    REQUIRE_PTR(v_out, "v_out", true);
    REQUIRE_PTR(workspace, "workspace", true);
    const WsLayout lay = layout_of(p);
    // every set holds at most N rows: no more can be asked of the kernels
    const long long cap = std::min((long long)capacity_rows, (long long)p.L * p.H_kv * p.N);
    cudaError_t e = launch_select_compact(p, scores, text_scores, budgets, modality, offsets, idx,
                                          k, v, k_out, v_out, cap, status_of(workspace, lay),
                                          static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "select/compact launch");
}

int tgvkv_select_compact_launches(const tgvkv_desc* desc) {
    Problem p{};
    if (make_problem(desc, &p)) return -1;
    return select_compact_launches(p);
}

int tgvkv_evict(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                const float* w, double ratio, float* scores, float* tvb_stat, int32_t* budgets,
                int64_t* offsets, int32_t* idx, uint16_t* k_out, uint16_t* v_out,
                void* workspace, void* stream) {
    return evict_impl(desc, q_text, k, v, modality, text_pos, w, ratio, false, nullptr, scores,
                      tvb_stat, budgets, offsets, idx, k_out, v_out, workspace, stream);
}

int tgvkv_evict_with_stats(const tgvkv_desc* desc, const uint16_t* q_text, const uint16_t* k,
                           const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                           const float* w, double ratio, const float* row_stats, float* scores,
                           float* tvb_stat, int32_t* budgets, int64_t* offsets, int32_t* idx,
                           uint16_t* k_out, uint16_t* v_out, void* workspace, void* stream) {
    return evict_impl(desc, q_text, k, v, modality, text_pos, w, ratio, true, row_stats, scores,
                      tvb_stat, budgets, offsets, idx, k_out, v_out, workspace, stream);
}

int tgvkv_prefill(const tgvkv_desc* desc, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                  const uint8_t* modality, const int32_t* text_pos, uint16_t* o, uint16_t* q_text,
                  float* row_stats, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    if ((long long)p.L * p.H_q * p.N >= (1LL << 31))
        return fail(TGVKV_ERR_UNSUPPORTED, "q holds 2^31 rows or more");
    REQUIRE_PTR(q, "q", true);
    REQUIRE_PTR(k, "k", true);
    REQUIRE_PTR(v, "v", true);
    REQUIRE_PTR(modality, "modality", false);
    REQUIRE_PTR(o, "o", true);
    if (p.n_win > 0) {
        REQUIRE_PTR(text_pos, "text_pos", false);
        REQUIRE_PTR(q_text, "q_text", true);
        REQUIRE_PTR(row_stats, "row_stats", false);
    }
    REQUIRE_PTR(workspace, "workspace", true);
    const WsLayout lay = layout_of(p);
    cudaError_t e = launch_prefill(p, q, k, v, modality, text_pos, o, q_text, row_stats,
                                   status_of(workspace, lay), static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "prefill launch");
}

int tgvkv_decode(const tgvkv_desc* desc, const uint16_t* q, const uint16_t* k_rows,
                 const uint16_t* v_rows, int64_t capacity_rows, const int64_t* offsets,
                 float* out, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    REQUIRE_PTR(q, "q", true);
    REQUIRE_PTR(k_rows, "k_rows", true);
    REQUIRE_PTR(v_rows, "v_rows", true);
    REQUIRE_PTR(offsets, "offsets", false);
    REQUIRE_PTR(out, "out", false);
    REQUIRE_PTR(workspace, "workspace", true);
    if (capacity_rows < 0)
        return fail(TGVKV_ERR_INVALID_ARG, "capacity_rows=%lld < 0", (long long)capacity_rows);
    if ((reinterpret_cast<uintptr_t>(offsets) & 7u) != 0)
        return fail(TGVKV_ERR_INVALID_ARG, "offsets is not 8-byte aligned");
    if ((reinterpret_cast<uintptr_t>(out) & 7u) != 0)
        return fail(TGVKV_ERR_INVALID_ARG, "out is not 8-byte aligned");
    const WsLayout lay = layout_of(p);
    char* ws = static_cast<char*>(workspace);
    cudaError_t e = launch_decode(p, q, k_rows, v_rows, (long long)capacity_rows, offsets, out,
                                  reinterpret_cast<float*>(ws + lay.decode_part),
                                  status_of(workspace, lay), static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "decode launch");
}

int tgvkv_check_wait_timeout(void* workspace, void* stream) {
    REQUIRE_PTR(workspace, "workspace", true);
    // the status word is the first word of every workspace layout
    cudaError_t e = launch_wait_timeout(static_cast<uint32_t*>(workspace),
                                        static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "wait-timeout launch");
}

int tgvkv_decode_launches(const tgvkv_desc* desc) {
    Problem p{};
    if (make_problem(desc, &p) != TGVKV_OK) return -1;
    return decode_launches(p);
}

int tgvkv_evict_launches(const tgvkv_desc* desc) {
    Problem p{};
    if (make_problem(desc, &p) != TGVKV_OK) return -1;
    const int text = needs_text_pass(p) ? score_launches(p) + (p.weights_eq7 && p.n_win > 0 ? 1 : 0) : 0;
    return text + (score_launches(p) == 0 ? 1 : score_launches(p)) + select_compact_launches(p);
}

int tgvkv_workspace_init(const tgvkv_desc* desc, void* workspace, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    REQUIRE_PTR(workspace, "workspace", true);
    cudaError_t e = cudaMemsetAsync(workspace, 0, layout_of(p).total, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ok() : cuda_fail(e, "workspace memset");
}

int tgvkv_status(void* workspace, void* stream) {
    if (!workspace) {
        fail(TGVKV_ERR_INVALID_ARG, "workspace is NULL");
        return -TGVKV_ERR_INVALID_ARG;
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint32_t bits = 0;
    // the status word sits at offset 0 of every workspace layout
    cudaError_t e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&bits, workspace, sizeof(bits), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(workspace, 0, sizeof(bits), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        cuda_fail(e, "status read");
        return -TGVKV_ERR_CUDA;
    }
    ok();
    return (int)bits;
}

const char* tgvkv_last_error(void) { return g_last_error; }

}  // extern "C"

// ---------------------------------------------------------------------------
// tgvkv_score_noalloc: tgvkv_score with its scratch in a fixed device array,
// for callers that receive only input/output buffers and may not allocate.
// ---------------------------------------------------------------------------
namespace {

// The scratch of every tgvkv_score_noalloc call on a device.  It keeps the
// previous call's contents; the call clears what must start at zero.
static __device__ __align__(256) unsigned char g_noalloc_scratch[TGVKV_NOALLOC_SCRATCH_BYTES];

// Device address of g_noalloc_scratch in the current device's context.  The
// name is a host-side stand-in: only this address may be given to a kernel.
// It is looked up on every call (a cheap query once the module is loaded), so
// a context created after cudaDeviceReset gets its own array's address.
int noalloc_scratch(void** out) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || ptr == nullptr)
        return tgvkv::cuda_fail(e, "cudaGetSymbolAddress(static scratch)");
    *out = ptr;
    return TGVKV_OK;
}

}  // namespace

extern "C" int tgvkv_score_noalloc(const tgvkv_desc* desc, const uint16_t* q_text,
                                   const uint16_t* k, const uint8_t* modality,
                                   const int32_t* text_pos, const float* w, float* scores,
                                   float* tvb_stat, void* stream) {
    Problem p{};
    int rc = make_problem(desc, &p);
    if (rc) return rc;
    const WsLayout lay = layout_of(p);
    if (lay.score_total > (size_t)TGVKV_NOALLOC_SCRATCH_BYTES)
        return fail(TGVKV_ERR_UNSUPPORTED,
                    "problem needs %zu bytes of scratch; the static scratch holds %u "
                    "(use tgvkv_score with a caller workspace)",
                    lay.score_total, (unsigned)TGVKV_NOALLOC_SCRATCH_BYTES);
    void* scratch = nullptr;
    if ((rc = noalloc_scratch(&scratch))) return rc;
    rc = check_score_args(p, q_text, k, modality, text_pos, w, scores, tvb_stat, scratch);
    if (rc) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the status word and the completion counters start at zero for every call
    cudaError_t e = cudaMemsetAsync(static_cast<char*>(scratch) + lay.status, 0, sizeof(uint32_t), st);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(static_cast<char*>(scratch) + lay.tickets, 0,
                            sizeof(uint32_t) * ticket_words(p), st);
    if (e != cudaSuccess) return cuda_fail(e, "static scratch clear");
    rc = do_score(p, q_text, k, modality, text_pos, w, scores, tvb_stat, scratch, st);
    return rc ? rc : ok();
}

extern "C" int tgvkv_noalloc_status(void* stream) {
    void* scratch = nullptr;
    int rc = noalloc_scratch(&scratch);
    if (rc) return -rc;
    // the status word sits at offset 0 of every workspace layout
    return tgvkv_status(scratch, stream);
}
