// Decode over the compacted cache (the consumer of the eviction step; the
// decode phase of Section 3.1): the new token's query of head h attends to the
// retained rows of KV head g = h / G,
//   o[l][h] = sum_r softmax_r(scale * <q, k_r>) v_r  over the rows r of set (l, g).
// A set without rows gives 0.
//
// HBM-bound: every retained K and V row is read once, so the kernel streams
// the rows of the CSR cache as one sequence.  One persistent CTA per SM; each
// of its warps is a row stream that takes one contiguous slice of
// [offsets[0], offsets[L*H_kv]) -- the same number of rows for every stream,
// whatever the set sizes -- and walks it in chunks of up to CH rows that never
// cross a set boundary.  A stream moves its chunks through its own two-stage
// ring of shared memory with TMA (K and V tiles of CH rows x 64 dims, 128-byte
// swizzle; a segment's last, partial chunk in 8-row boxes; the pass's 8 query
// rows with a segment's first chunk), so every stream keeps two chunks in
// flight and never waits for another.
//
// Arithmetic on the tensor cores (mma.sync m16n8k16: bf16 operands, fp32
// accumulation), per chunk and for up to 8 query heads of the group at a time:
//   S = Q K^T   rows 0-7 of the 16-row operand are the heads, rows 8-15 zero;
//   O += P V    rows 0-7 carry bf16(P) and rows 8-15 the remainder
//               bf16(P - bf16(P)), so the two halves together keep P to about
//               16 bits (a plain bf16 P would move an output by ~1e-3).
// The softmax is online, in base 2.  A set that one stream covers whole is
// written out directly; a set split over several streams leaves one partial
// (m, l, O) per stream, and a second kernel, launched as a programmatic
// dependent of the first (its launch overlaps the first kernel's tail), merges
// them: one warp per (set, query head), the partials in stream order, so the
// result does not depend on timing.  The second kernel also checks the CSR
// and writes 0 for empty sets.  Groups of more than 8 query heads take
// several passes (blockIdx.y), each over all rows.
#include <cuda_bf16.h>

#include "common.cuh"
#include "launch.h"
#include "tc05.cuh"

namespace tgvkv {
namespace {

constexpr int kDecStages = 2;         // chunks in flight per stream
constexpr int kDecHeads = 8;          // query heads per pass
constexpr int kDecOffsCache = 4096;   // offsets entries kept in shared memory

template <int D, int CH, int W>
struct DecGeom {
    static constexpr int KT = D / 64;                       // 64-dim tiles of a row
    static constexpr int kTile = CH * 128;                  // bytes: one 64-dim tile of a chunk
    static constexpr int kQTile = kDecHeads * 128;          // bytes: one 64-dim tile of 8 query rows
    static constexpr int kK = 0;                            // offsets inside a stage
    static constexpr int kV = KT * kTile;
    static constexpr int kQ = 2 * KT * kTile;
    static constexpr int kStage = 2 * KT * kTile + KT * kQTile;
    static constexpr int kRing = W * kDecStages * kStage;
    static_assert(CH == 16 || CH == 32, "chunk rows");
};

// One chunk of a stream: rows [r0, r0 + n) of set s.
struct DecChunk {
    int r0, s, n;
    int first, last;   // the first / last chunk of the stream's segment of set s
};

// Shared memory after the rings (which start 1024-byte aligned).
template <int W>
struct DecTail {
    uint64_t full[W][kDecStages];
    DecChunk chunk[W][kDecStages];
};

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

// c += A B over one 16 x 8 x 16 tile (A row-major, B column-major, bf16; c fp32).
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Byte offset of 16-byte unit u (0..7) of row r in a tile written by TMA with
// the 128-byte swizzle (tile base 1024-byte aligned).
__device__ __forceinline__ uint32_t swz(int r, int u) {
    return (uint32_t)(r * 128 + ((u ^ (r & 7)) << 4));
}

// Two floats as bf16x2, `lo` in the low half (the operand element of the
// lower column index).
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ int clampi(long long x, int lo, int hi) {
    return x < lo ? lo : (x > hi ? hi : (int)x);
}

// The CSR offsets, each clipped to [0, cap]: from shared memory when they fit
// there, else read from global memory and clipped on the way.
struct DecRows {
    const int* so;
    const long long* go;
    int cap, R0, R1;
    bool cached;
    __device__ __forceinline__ int at(int i) const { return cached ? so[i] : clampi(go[i], 0, cap); }
    // rows of set s, clipped to the rows the kernel reads, [R0, R1)
    __device__ __forceinline__ void of(int s, int& lo, int& hi) const {
        lo = min(max(at(s), R0), R1);
        hi = min(max(at(s + 1), lo), R1);
    }
};

// The largest s in [0, n_sets) with offset s <= a (0 if none).
__device__ __forceinline__ int dec_find_set(const DecRows& rows, int n_sets, int a) {
    int lo = 0, hi = n_sets - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (rows.at(mid) <= a) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

// A stream's walk over its rows [a, end): set by set, CH rows at a time.
template <int CH>
struct DecWalk {
    int r, e, seg0, a, end, s;

    __device__ __forceinline__ void init(const DecRows& rows, int n_sets, int a_, int end_) {
        a = a_;
        end = end_;
        s = dec_find_set(rows, n_sets, a);
        int lo, hi;
        rows.of(s, lo, hi);
        seg0 = r = max(lo, a);
        e = min(hi, end);
    }

    __device__ __forceinline__ bool next(const DecRows& rows, int n_sets, DecChunk& c) {
        while (r >= e) {
            if (++s >= n_sets) return false;
            int lo, hi;
            rows.of(s, lo, hi);
            seg0 = r = max(lo, a);
            e = min(hi, end);
            if (r >= end) return false;
        }
        c.r0 = r;
        c.s = s;
        c.n = min(e - r, CH);
        c.first = r == seg0;
        c.last = r + c.n == e;
        r += c.n;
        return true;
    }
};

// Lane 0 of a stream: the TMA loads of chunk c into one stage of its ring.
// Full chunks move as CH-row boxes; a shorter one as ceil(n / 8) 8-row boxes
// (rows past n belong to the next set or lie past the cache: loaded, or
// zero-filled, and masked).  A segment's first chunk also brings the 8 query
// rows of the pass (rows past the group's heads are other heads' rows or
// zero-filled, and never written out).
template <int D, int CH, int W>
__device__ __forceinline__ void dec_issue(unsigned char* stage, uint64_t* bar, const DecChunk& c,
                                          const CUtensorMap* mkf, const CUtensorMap* mk8,
                                          const CUtensorMap* mvf, const CUtensorMap* mv8,
                                          const CUtensorMap* mq, const Problem& p, int hb) {
    using Gm = DecGeom<D, CH, W>;
    const int nb8 = c.n == CH ? 0 : (c.n + 7) >> 3;
    const uint32_t kv = nb8 ? (uint32_t)nb8 * 1024u : (uint32_t)Gm::kTile;
    const uint32_t bytes = 2u * Gm::KT * kv + (c.first ? (uint32_t)(Gm::KT * Gm::kQTile) : 0u);
    tc::mbar_arrive_expect_tx(bar, bytes);
#pragma unroll
    for (int kt = 0; kt < Gm::KT; ++kt) {
        if (!nb8) {
            tc::tma_load_2d(stage + Gm::kK + kt * Gm::kTile, mkf, 64 * kt, c.r0, bar);
            tc::tma_load_2d(stage + Gm::kV + kt * Gm::kTile, mvf, 64 * kt, c.r0, bar);
        } else {
            for (int b = 0; b < nb8; ++b) {
                tc::tma_load_2d(stage + Gm::kK + kt * Gm::kTile + b * 1024, mk8, 64 * kt, c.r0 + 8 * b,
                                bar);
                tc::tma_load_2d(stage + Gm::kV + kt * Gm::kTile + b * 1024, mv8, 64 * kt, c.r0 + 8 * b,
                                bar);
            }
        }
    }
    if (c.first) {
        const int l = c.s / p.H_kv, g = c.s % p.H_kv;
        const int qrow = l * p.H_q + g * p.G + hb * kDecHeads;
#pragma unroll
        for (int kt = 0; kt < Gm::KT; ++kt)
            tc::tma_load_2d(stage + Gm::kQ + kt * Gm::kQTile, mq, 64 * kt, qrow, bar);
    }
}

// Partial result of stream w, slot 0 (the segment that starts the stream's
// rows) or 1 (the one that ends them): O [hpp][D], m [hpp], l [hpp].
__device__ __forceinline__ float* dec_slot(float* part, int n_streams, int hb, int w, int slot,
                                           int rec) {
    return part + (((size_t)hb * n_streams + w) * 2 + slot) * (size_t)rec;
}

template <int D, int CH, int W>
__global__ void __launch_bounds__(W * 32, 1)
decode_kernel(const __grid_constant__ CUtensorMap mkf, const __grid_constant__ CUtensorMap mk8,
              const __grid_constant__ CUtensorMap mvf, const __grid_constant__ CUtensorMap mv8,
              const __grid_constant__ CUtensorMap mq, const Problem p,
              const int64_t* __restrict__ offsets, int cap, float* __restrict__ out,
              float* __restrict__ part, uint32_t* __restrict__ status) {
    using Gm = DecGeom<D, CH, W>;
    // the merge kernel may be scheduled now; it waits for this grid's results
    griddep_launch_dependents();
    if (threadIdx.x == 0) {   // the descriptors' first fetch overlaps the prologue
        tc::tma_prefetch_desc(&mkf);
        tc::tma_prefetch_desc(&mk8);
        tc::tma_prefetch_desc(&mvf);
        tc::tma_prefetch_desc(&mv8);
        tc::tma_prefetch_desc(&mq);
    }
    constexpr int KS = D / 16;    // 16-dim steps of S = Q K^T
    constexpr int ND = D / 8;     // 8-dim column tiles of O
    constexpr int NT = CH / 8;    // 8-key column tiles of S
    constexpr int KK = CH / 16;   // 16-key steps of O += P V
    extern __shared__ unsigned char dec_smem_raw[];
    unsigned char* ring = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dec_smem_raw) + 1023) & ~uintptr_t(1023));
    DecTail<W>& tl = *reinterpret_cast<DecTail<W>*>(ring + Gm::kRing);
    int* offs_s = reinterpret_cast<int*>(&tl + 1);
    __shared__ int never;   // the waits' abort flag: streams never abort one another

    const int n_sets = p.L * p.H_kv;
    const int hb = blockIdx.y;
    const int nh = min(kDecHeads, p.G - hb * kDecHeads);
    const int hpp = decode_heads(p), rec = decode_record_floats(p);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    DecRows rows;
    rows.so = offs_s;
    rows.go = reinterpret_cast<const long long*>(offsets);
    rows.cap = cap;
    rows.cached = n_sets + 1 <= kDecOffsCache;
    if (rows.cached) {
        // all loads first, then the stores: one round trip for up to 8 entries a thread
        for (int b = 0; b <= n_sets; b += 8 * W * 32) {
            long long v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int idx = b + u * W * 32 + tid;
                v[u] = idx <= n_sets ? rows.go[idx] : 0;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int idx = b + u * W * 32 + tid;
                if (idx <= n_sets) offs_s[idx] = clampi(v[u], 0, cap);
            }
        }
    }
    // Zero the rings once: the rows of a k-step that no box of a short chunk
    // loads then hold zeros or rows of an earlier chunk, never stale bits.
    for (int i = tid; i < Gm::kRing / 16; i += blockDim.x)
        reinterpret_cast<uint4*>(ring)[i] = make_uint4(0u, 0u, 0u, 0u);
    if (tid == 0) never = 0;
    if (lane == 0) {
        for (int st = 0; st < kDecStages; ++st) tc::mbar_init(&tl.full[warp][st], 1);
        tc::fence_mbar_init();
    }
    fence_proxy_async();   // the zeroed rings before any TMA write to them
    __syncthreads();

    rows.R0 = rows.at(0);
    rows.R1 = max(rows.at(n_sets), rows.R0);
    const int n_streams = gridDim.x * W;
    const int per = (int)(((long long)rows.R1 - rows.R0 + n_streams - 1) / n_streams);
    const int si = blockIdx.x * W + warp;
    const int a = rows.R0 + (int)min((long long)si * per, (long long)rows.R1 - rows.R0);
    const int end = rows.R0 + (int)min((long long)(si + 1) * per, (long long)rows.R1 - rows.R0);

    // the stream's first chunks
    unsigned char* wring = ring + warp * kDecStages * Gm::kStage;
    DecWalk<CH> walk;
    int issued = 0;
    if (a < end) {
        walk.init(rows, n_sets, a, end);
        for (int st = 0; st < kDecStages; ++st) {
            DecChunk c;
            if (!walk.next(rows, n_sets, c)) break;
            if (lane == 0) {
                tl.chunk[warp][st] = c;
                dec_issue<D, CH, W>(wring + st * Gm::kStage, &tl.full[warp][st], c, &mkf, &mk8, &mvf,
                                    &mv8, &mq, p, hb);
            }
            ++issued;
        }
    }
    __syncwarp();
    if (issued == 0) return;

    const int g = lane >> 2, tq = lane & 3;   // MMA fragment row (head) and column pair
    uint32_t qa[KS][2];                       // Q fragments (rows 0-7), per 16-dim step
    float o[ND][4];                           // O: rows g (bf16(P) part) and g + 8 (remainder)
    float m = -INFINITY, lsum = 0.f;
    int seg_start = 0;
#pragma unroll
    for (int nd = 0; nd < ND; ++nd)
#pragma unroll
        for (int e = 0; e < 4; ++e) o[nd][e] = 0.f;
#pragma unroll
    for (int k = 0; k < KS; ++k) qa[k][0] = qa[k][1] = 0u;

    int i = 0;
    for (; i < issued; ++i) {
        const int st = i % kDecStages;
        const bool got = tc::mbar_wait(&tl.full[warp][st], (i / kDecStages) & 1, &never);
        if (!__all_sync(~0u, got)) break;
        const DecChunk c = tl.chunk[warp][st];
        const uint32_t sb = smem_u32(wring + st * Gm::kStage);
        if (c.first) {
            seg_start = c.r0;
#pragma unroll
            for (int u2 = 0; u2 < KS / 2; ++u2) {
                const int unit = 4 * u2 + (lane >> 3);
                uint32_t r[4];
                ldsm_x4(sb + Gm::kQ + (unit >> 3) * Gm::kQTile + swz(lane & 7, unit & 7), r);
                qa[2 * u2][0] = r[0];
                qa[2 * u2][1] = r[1];
                qa[2 * u2 + 1][0] = r[2];
                qa[2 * u2 + 1][1] = r[3];
            }
            m = -INFINITY;
            lsum = 0.f;
#pragma unroll
            for (int nd = 0; nd < ND; ++nd)
#pragma unroll
                for (int e = 0; e < 4; ++e) o[nd][e] = 0.f;
        }
        // S = Q K^T over the chunk's keys; n-tile j holds keys 8j..8j+7.  Two
        // accumulators per tile (alternate 32-dim blocks) halve the MMA chains.
        float sacc[2][NT][4];
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int j = 0; j < NT; ++j)
#pragma unroll
                for (int e = 0; e < 4; ++e) sacc[h][j][e] = 0.f;
#pragma unroll
        for (int u2 = 0; u2 < KS / 2; ++u2) {
            const int unit = 4 * u2 + (lane >> 3);
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                const int row = 8 * j + (lane & 7);
                uint32_t r[4];
                ldsm_x4(sb + Gm::kK + (unit >> 3) * Gm::kTile + swz(row, unit & 7), r);
                mma_bf16(sacc[u2 & 1][j], qa[2 * u2][0], 0u, qa[2 * u2][1], 0u, r[0], r[1]);
                mma_bf16(sacc[u2 & 1][j], qa[2 * u2 + 1][0], 0u, qa[2 * u2 + 1][1], 0u, r[2], r[3]);
            }
        }
        // online softmax of head g over the chunk (the 4 lanes of a head share it)
        float sv[2 * NT];
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int e = 0; e < 2; ++e)
                sv[2 * j + e] = 8 * j + 2 * tq + e < c.n
                                    ? (sacc[0][j][e] + sacc[1][j][e]) * p.scale_log2
                                    : -INFINITY;
        float cm = sv[0];
#pragma unroll
        for (int k = 1; k < 2 * NT; ++k) cm = fmaxf(cm, sv[k]);
        cm = fmaxf(cm, __shfl_xor_sync(~0u, cm, 1));
        cm = fmaxf(cm, __shfl_xor_sync(~0u, cm, 2));
        const float mn = fmaxf(m, cm);
        const float alpha = fast_exp2(m - mn);   // m = -inf (first chunk): 0
        float pr[2 * NT], ps = 0.f;
#pragma unroll
        for (int k = 0; k < 2 * NT; ++k) {
            pr[k] = fast_exp2(sv[k] - mn);
            ps += pr[k];
        }
        lsum = lsum * alpha + ps;
        m = mn;
        if (__any_sync(~0u, alpha != 1.f)) {   // the running maximum moved for some head
#pragma unroll
            for (int nd = 0; nd < ND; ++nd)
#pragma unroll
                for (int e = 0; e < 4; ++e) o[nd][e] *= alpha;
        }
        // O += P V: 16-key steps kk (n-tiles 2kk and 2kk + 1 of S)
#pragma unroll
        for (int kk = 0; kk < KK; ++kk) {
            if (16 * kk >= c.n) break;
            const uint32_t h01 = pack_bf16(pr[4 * kk], pr[4 * kk + 1]);
            const uint32_t h23 = pack_bf16(pr[4 * kk + 2], pr[4 * kk + 3]);
            const uint32_t l01 = pack_bf16(pr[4 * kk] - __uint_as_float(h01 << 16),
                                           pr[4 * kk + 1] - __uint_as_float(h01 & 0xFFFF0000u));
            const uint32_t l23 = pack_bf16(pr[4 * kk + 2] - __uint_as_float(h23 << 16),
                                           pr[4 * kk + 3] - __uint_as_float(h23 & 0xFFFF0000u));
            const int row = 16 * kk + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
            for (int nd2 = 0; nd2 < ND / 2; ++nd2) {
                const int unit = 2 * nd2 + (lane >> 4);
                uint32_t r[4];
                ldsm_x4_trans(sb + Gm::kV + (unit >> 3) * Gm::kTile + swz(row, unit & 7), r);
                mma_bf16(o[2 * nd2], h01, l01, h23, l23, r[0], r[1]);
                mma_bf16(o[2 * nd2 + 1], h01, l01, h23, l23, r[2], r[3]);
            }
        }
        // the stage is read: refill it with the stream's next chunk
        __syncwarp();
        {
            DecChunk nc;
            if (walk.next(rows, n_sets, nc)) {
                if (lane == 0) {
                    tl.chunk[warp][st] = nc;
                    dec_issue<D, CH, W>(wring + st * Gm::kStage, &tl.full[warp][st], nc, &mkf, &mk8,
                                        &mvf, &mv8, &mq, p, hb);
                }
                ++issued;
            }
        }
        if (!c.last) continue;
        // ---- the stream's segment of set c.s is complete
        float lt = lsum;
        lt += __shfl_xor_sync(~0u, lt, 1);
        lt += __shfl_xor_sync(~0u, lt, 2);
        int lo, hi;
        rows.of(c.s, lo, hi);
        const int w0 = (lo - rows.R0) / per, w1 = (hi - 1 - rows.R0) / per;
        const int l = c.s / p.H_kv, gk = c.s % p.H_kv;
        float* out_head0 = out + ((size_t)l * p.H_q + gk * p.G + hb * kDecHeads) * D;
        if (w0 == w1) {   // the set lies inside this stream
            if (g < nh) {
                const float inv = lt > 0.f ? 1.f / lt : 0.f;
                float* op = out_head0 + g * D + 2 * tq;
#pragma unroll
                for (int nd = 0; nd < ND; ++nd)
                    *reinterpret_cast<float2*>(op + 8 * nd) =
                        make_float2((o[nd][0] + o[nd][2]) * inv, (o[nd][1] + o[nd][3]) * inv);
            }
            continue;
        }
        // a split set: this stream's partial result (slot 0: the segment the
        // stream starts with, 1: the one it ends with), merged by the second kernel
        float* pp = dec_slot(part, n_streams, hb, si, seg_start == a ? 0 : 1, rec);
        if (g < hpp) {
            float* op = pp + g * D + 2 * tq;
#pragma unroll
            for (int nd = 0; nd < ND; ++nd)
                *reinterpret_cast<float2*>(op + 8 * nd) =
                    make_float2(o[nd][0] + o[nd][2], o[nd][1] + o[nd][3]);
            if (tq == 0) {
                pp[hpp * D + g] = m;
                pp[hpp * D + hpp + g] = lt;
            }
        }
    }
    if (i < issued) {
        // a wait gave up: report it, and give the copies still in flight into
        // this stream's ring a bounded time to land before the CTA exits
        if (lane == 0) raise_status(status, TGVKV_STATUS_TIMEOUT);
        for (; i < issued; ++i)
            if (!tc::mbar_wait(&tl.full[warp][i % kDecStages], (i / kDecStages) & 1, &never)) break;
    }
}

// The split sets' merge, the CSR check and the empty sets: one warp per
// (set, query head of the pass).  Launched as a programmatic dependent of
// decode_kernel: it reads its inputs, then waits for that grid's partial
// results.  A split set's partials are combined in stream order: the lanes
// fetch the streams' (m, l) side by side, so the common maximum and every
// weight cost one round trip; then lane t adds dims [t * D/32, (t+1) * D/32)
// of the weighted O of each stream, loading 8 streams' values at a time.
template <int D>
__global__ void __launch_bounds__(128)
decode_merge_kernel(const Problem p, const int64_t* __restrict__ offsets, int cap, int n_streams,
                    const float* __restrict__ part, float* __restrict__ out,
                    uint32_t* __restrict__ status) {
    constexpr int DPL = D / 32;
    const int lane = threadIdx.x & 31;
    const int n_sets = p.L * p.H_kv;
    const int hb = blockIdx.y;
    const int nh = min(kDecHeads, p.G - hb * kDecHeads);
    const int hpp = decode_heads(p), rec = decode_record_floats(p);
    const int gw = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int s = gw / hpp, hh = gw % hpp;
    // inputs only before the wait (the first kernel writes none of them); its
    // partial results after it, through L2
    long long lo_raw = 0, hi_raw = 0, r0_raw = 0, r1_raw = 0;
    if (s < n_sets) {
        lo_raw = offsets[s];
        hi_raw = offsets[s + 1];
        r0_raw = offsets[0];
        r1_raw = offsets[n_sets];
    }
    griddep_wait();
    if (s >= n_sets || hh >= nh) return;
    // every set's rows must lie in order inside [0, cap)
    if (hh == 0 && lane == 0 && (lo_raw < 0 || hi_raw < lo_raw || hi_raw > cap))
        raise_status(status, TGVKV_STATUS_INDEX);
    // the first kernel's clipping and split of the rows
    const int R0 = clampi(r0_raw, 0, cap), R1 = max(clampi(r1_raw, 0, cap), R0);
    const int lo = min(max(clampi(lo_raw, 0, cap), R0), R1);
    const int hi = min(max(clampi(hi_raw, 0, cap), lo), R1);
    const int l = s / p.H_kv, gk = s % p.H_kv;
    float* o = out + ((size_t)l * p.H_q + gk * p.G + hb * kDecHeads + hh) * D + DPL * lane;
    if (hi <= lo) {   // an empty set gives 0
#pragma unroll
        for (int c = 0; c < DPL; ++c) o[c] = 0.f;
        return;
    }
    const int per = (int)(((long long)R1 - R0 + n_streams - 1) / n_streams);
    const int w0 = (lo - R0) / per, w1 = (hi - 1 - R0) / per;
    if (w0 == w1) return;   // inside one stream: written by the first kernel
    const bool w0_second = lo != R0 + w0 * per;
    const int nw = w1 - w0 + 1;
    auto slot_of = [&](int w) {
        return dec_slot(const_cast<float*>(part), n_streams, hb, w, (w == w0 && w0_second) ? 1 : 0,
                        rec);
    };
    float Lt = 0.f, acc[DPL];
#pragma unroll
    for (int c = 0; c < DPL; ++c) acc[c] = 0.f;
    float M = -INFINITY;
    for (int b = 0; b < nw; b += 32) {
        // (m, l) of 32 streams side by side: the common maximum and the weights
        // in one round trip (a later batch of 32 rescales what came before)
        const int cnt = nw - b < 32 ? nw - b : 32;
        float mw = -INFINITY, lw = 0.f;
        if (lane < cnt) {
            const float* pp = slot_of(w0 + b + lane);
            mw = __ldcg(pp + hpp * D + hh);
            lw = __ldcg(pp + hpp * D + hpp + hh);
        }
        float Mb = mw;
#pragma unroll
        for (int k = 16; k > 0; k >>= 1) Mb = fmaxf(Mb, __shfl_xor_sync(~0u, Mb, k));
        const float Mn = fmaxf(M, Mb);
        if (!(Mn > -INFINITY)) continue;   // no mass yet
        const float fa = fast_exp2(M - Mn);   // M = -inf: 0
        // a segment without mass (m = -inf) adds nothing
        const float f = mw > -INFINITY ? fast_exp2(mw - Mn) : 0.f;
        float lf = lw * f;
#pragma unroll
        for (int k = 16; k > 0; k >>= 1) lf += __shfl_xor_sync(~0u, lf, k);
        Lt = Lt * fa + lf;
#pragma unroll
        for (int c = 0; c < DPL; ++c) acc[c] *= fa;
        M = Mn;
        // the weighted O of the batch, 8 streams' loads in flight at a time
        for (int j0 = 0; j0 < cnt; j0 += 8) {
            float ov[8][DPL];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                if (j0 + u < cnt) {
                    const float* ow = slot_of(w0 + b + j0 + u) + hh * D + DPL * lane;
                    if (DPL == 4) {
                        const float4 t = __ldcg(reinterpret_cast<const float4*>(ow));
                        ov[u][0] = t.x;
                        ov[u][1 % DPL] = t.y;
                        ov[u][2 % DPL] = t.z;
                        ov[u][3 % DPL] = t.w;
                    } else {
                        const float2 t = __ldcg(reinterpret_cast<const float2*>(ow));
                        ov[u][0] = t.x;
                        ov[u][1 % DPL] = t.y;
                    }
                } else {
#pragma unroll
                    for (int c = 0; c < DPL; ++c) ov[u][c] = 0.f;
                }
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const float fj = __shfl_sync(~0u, f, (j0 + u) & 31);
#pragma unroll
                for (int c = 0; c < DPL; ++c) acc[c] += ov[u][c] * fj;
            }
        }
    }
    const float inv = Lt > 0.f ? 1.f / Lt : 0.f;
#pragma unroll
    for (int c = 0; c < DPL; ++c) o[c] = acc[c] * inv;
}

// Rows per chunk and streams (warps) per CTA.
constexpr int kDecCH = 16;
constexpr int kDecW = 8;

template <int D, int CH, int W>
cudaError_t launch_dec(const Problem& p, const uint16_t* q, const uint16_t* k_rows,
                       const uint16_t* v_rows, long long capacity_rows, const int64_t* offsets,
                       float* out, float* part, uint32_t* status, cudaStream_t stream) {
    using Gm = DecGeom<D, CH, W>;
    // TMA row coordinates are 32-bit: rows from 2^31 - 1 on are never read (a
    // CSR that reaches them reports TGVKV_STATUS_INDEX)
    const int cap = capacity_rows > 0x7FFFFFFFll ? 0x7FFFFFFF : (int)capacity_rows;
    const uint64_t map_rows = cap > 0 ? (uint64_t)cap : 1u;   // no row is read when cap = 0
    alignas(64) CUtensorMap mkf, mk8, mvf, mv8, mq;
    if (!make_tile_map(&mkf, k_rows, map_rows, D, CH) ||
        !make_tile_map(&mk8, k_rows, map_rows, D, 8) ||
        !make_tile_map(&mvf, v_rows, map_rows, D, CH) ||
        !make_tile_map(&mv8, v_rows, map_rows, D, 8) ||
        !make_tile_map(&mq, q, (uint64_t)p.L * p.H_q, D, kDecHeads))
        return cudaErrorInvalidValue;
    const int n_sets = p.L * p.H_kv;
    const size_t offs_bytes = n_sets + 1 <= kDecOffsCache ? sizeof(int) * (n_sets + 1) : 0;
    const size_t smem = 1024 + Gm::kRing + sizeof(DecTail<W>) + offs_bytes;
    static_assert(1024 + Gm::kRing + sizeof(DecTail<W>) + sizeof(int) * kDecOffsCache <= 227 * 1024,
                  "shared memory of one CTA");
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<D, CH, W>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int sms = device_sm_count();
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int ctas = sms < kDecMaxStreams / W ? sms : kDecMaxStreams / W;
    decode_kernel<D, CH, W><<<dim3(ctas, decode_passes(p)), W * 32, smem, stream>>>(
        mkf, mk8, mvf, mv8, mq, p, offsets, cap, out, part, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // the merge, as a programmatic dependent: it is scheduled while the first
    // kernel runs and waits on the device for its results
    const long long warps = (long long)n_sets * decode_heads(p);
    return launch_dependent(decode_merge_kernel<D>, dim3((unsigned)((warps + 3) / 4), decode_passes(p)),
                            dim3(128), 0, stream, p, offsets, cap, ctas * W,
                            static_cast<const float*>(part), out, status);
}

}  // namespace

cudaError_t launch_decode(const Problem& p, const uint16_t* q, const uint16_t* k_rows,
                          const uint16_t* v_rows, long long capacity_rows, const int64_t* offsets,
                          float* out, float* part, uint32_t* status, cudaStream_t stream) {
    if (p.d == 64)
        return launch_dec<64, kDecCH, kDecW>(p, q, k_rows, v_rows, capacity_rows, offsets, out,
                                             part, status, stream);
    return launch_dec<128, kDecCH, kDecW>(p, q, k_rows, v_rows, capacity_rows, offsets, out, part,
                                          status, stream);
}

int decode_launches(const Problem&) { return 2; }

}  // namespace tgvkv
