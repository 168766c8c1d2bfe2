// Device-side helpers shared by the TGV-KV kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "tgvkv.h"

namespace tgvkv {

// Problem as the kernels see it.  Built on the host from tgvkv_desc.
struct Problem {
    int L, H_q, H_kv, G, d, N, N_v, N_t, n_win;
    int R;                 // query rows per KV head: G * n_win
    int T;                 // 128-row tiles per KV head: ceil(R / 128)
    float scale_log2;      // softmax_scale * log2(e): logits in base-2 units
    long long w_stride;    // floats between the weight rows of two layers
    int basis;             // TGVKV_BASIS_VISION or TGVKV_BASIS_ALL
    int weights_eq7;       // tgvkv_evict derives w~ by Eq. 7
    int keep_first, keep_last;   // sink tokens, clipped to [0, N]
    int budget_stat;       // statistic the budgets split: TGVKV_STAT_TV / _TT / _UNIFORM
    int head_budgets;      // one budget per (layer, KV head) instead of per layer
    // Score kernel only: the key set of pass B.  0 = vision keys (Eq. 8, row
    // weights w~); 1 = text keys with unit row weights (Eq. 9).  N_v then
    // holds the size of that key set, N_t; the launcher sets both.
    int keys_text;
    // Row statistics (m, Z, vision mass) per global query row, float [3 * L*H_q*n_win]:
    // the text-key pass writes them when not null; with stats_given the vision
    // pass reads them and skips its pass A (tgvkv_evict with a text-key pass).
    float* row_stats;
    int stats_given;
};

// Decode (decode.cu): at most kDecMaxStreams row streams (warps; one CTA per
// SM); a stream leaves at most two partial results of decode_heads(p) query
// heads x (d + 2) floats per pass over the rows, a pass taking up to 8 query
// heads of a group.
constexpr int kDecMaxStreams = 2048;
__host__ __device__ inline int decode_passes(const Problem& p) { return (p.G + 7) / 8; }
__host__ __device__ inline int decode_heads(const Problem& p) { return p.G < 8 ? p.G : 8; }
// floats of one partial result: O [heads][d], then m [heads] and l [heads],
// padded to a multiple of 4 floats (16-byte aligned records)
__host__ __device__ inline int decode_record_floats(const Problem& p) {
    return decode_heads(p) * p.d + ((2 * decode_heads(p) + 3) & ~3);
}

// Sinks among the positions 0..N-1: the first keep_first and the last keep_last.
__host__ __device__ inline bool is_sink(const Problem& p, int j) {
    return j < p.keep_first || j >= p.N - p.keep_last;
}

// Workspace layout (byte offsets into the caller's buffer).
struct WsLayout {
    size_t status;      // uint32 status word
    size_t tickets;     // uint32 [ticket_words]: completion counters (heads), kernel counters
    size_t stat_part;   // float [L*H_kv*T]: TV mass of one row tile
    size_t stat_head;   // float [L*H_kv]: TV mass of one KV head
    size_t score_part;  // float [L*H_kv*T*max(N_v,N_t)]: scores of one row tile (T > 1)
    // tgvkv_evict with Eq. 7 weights or the all-token basis only (0 otherwise):
    size_t text_scores; // float [L*H_kv*N_t]: Eq. 9 scores
    size_t weights;     // float [L*n_win]: Eq. 7 weights
    size_t stat_text;   // float [L]: the text-key pass's (unused) statistic
    size_t row_stats;   // float [3*L*H_q*n_win]: per-row (m, Z, vision mass) of the text-key pass
    size_t score_total; // bytes of everything above: what tgvkv_score / tgvkv_evict use
    // tgvkv_decode only (after score_total):
    size_t decode_part; // float [passes*kDecMaxStreams*2*record]: partials of split sets
    size_t total;
};

// Work items of one KV head in the score kernel: pairs of 128-row tiles
// (P = ceil(T / 2)) when the head has more than one row tile, else 1.
__host__ __device__ inline int score_pairs(const Problem& p) {
    return p.T >= 2 ? (p.T + 1) / 2 : 1;
}

// Counters at the start of the workspace: one per KV head, then the score
// kernel's work counter, the count of CTAs that ran out of work, and the count
// of CTAs that finished.
__host__ __device__ inline size_t ticket_words(const Problem& p) {
    return (size_t)p.L * p.H_kv + 3;
}

constexpr int kMaxN = 32768;     // key positions per head (the per-CTA tile maps)
constexpr int kMaxNv = 49152;    // vision keys held in shared memory by select
constexpr int kMaxL = 1024;      // layers handled by the budget kernel

// Programmatic dependent launch: a kernel launched with the programmatic
// stream-serialization attribute may start while the kernel before it on the
// stream runs; griddep_wait blocks until that kernel has completed (a no-op
// for an ordinary launch).  What that kernel wrote must then be read through
// L2 (__ldcg), not the read-only path: a dependent that started early can
// otherwise read a recycled buffer's old contents.  A kernel that calls
// griddep_launch_dependents lets its dependent be scheduled from then on.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void raise_status(uint32_t* status, uint32_t bits) {
    atomicOr(status, bits);
}

// 2^x with the MUFU.EX2 unit (PTX ex2.approx.ftz.f32; ex2(-inf) = +0).
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// log2(x) with the MUFU.LG2 unit (PTX lg2.approx.ftz.f32; lg2(0) = -inf).
__device__ __forceinline__ float fast_log2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Packed pairs of fp32 (Blackwell f32x2 FMA-pipe instructions).
union F2 {
    float2 f;
    unsigned long long u;
};
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    F2 x, y, z, r;
    x.f = a; y.f = b; z.f = c;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r.u) : "l"(x.u), "l"(y.u), "l"(z.u));
    return r.f;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    F2 x, y, r;
    x.f = a; y.f = b;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r.u) : "l"(x.u), "l"(y.u));
    return r.f;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Order-preserving map of an fp32 value to uint32 (larger float -> larger key).
__device__ __forceinline__ uint32_t float_order_key(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

}  // namespace tgvkv
