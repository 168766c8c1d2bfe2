// Causal prefill attention on the 5th-generation tensor cores (tcgen05) that
// also keeps what the eviction step needs from the rows at its query
// positions, so that the step's own pass over the row statistics goes away.
//
// Every token i of every (layer l, query head h) attends to the keys j <= i of
// its KV head g = h / G (Eq. 2 over all N rows):
//
//     o_i = sum_{j <= i} softmax_j(scale <q_i, k_j>) v_j
//
// A work item is one 128-row tile t of one (layer, query head); a persistent
// CTA takes items t-major, longest causal range first.  It streams the head's
// K and V tiles 0..t through one TMA ring, in the order the tensor core uses
// them: K_0, K_1, V_0, K_2, V_1, ...
//
//   S_j = Q K_j^T            TMEM, two 128-column buffers, alternating
//   softmax warps (thread = row): row maximum, P_j = 2^(x sl2 - m) rounded to
//            bf16 into shared memory, running normaliser l and vision mass;
//            O is rescaled only when a row's maximum rises more than 2^8 above
//            the reference m it uses (m then moves up to the new maximum)
//   O += P_j V_j             TMEM, D columns; V is the MN-major operand
//
// MMA order QK_0, QK_1, PV_0, QK_2, PV_1, ...: the softmax of tile j overlaps
// PV_{j-1} and QK_{j+1}.
//
// At the rows whose position is one of the eviction step's query positions
// (text_pos) the epilogue writes (m, Z, V): the row's reference maximum in
// base-2 units (logit x log2 e), Z = sum_j 2^(x_ij sl2 - m) and the same sum
// over the vision keys (Eq. 6's slice), and copies the row's query to q_text.
// The eviction's score passes read them instead of computing them (Eq. 2, 5,
// 6): the prefill already streams every key of those rows.
//
// Roles: warp 0 issues the TMA loads, warp 1 the MMAs (and owns the TMEM),
// warps 2-5 run the softmax, one per TMEM lane quarter, warp 6 copies the
// query rows to q_text.  Every wait is bounded
// (about 1 s of SM cycles); a timeout sets TGVKV_STATUS_TIMEOUT and the CTA
// unwinds after its copies and MMAs have finished.
#include <cuda_bf16.h>
#include <limits.h>
#include <math.h>

#include "common.cuh"
#include "launch.h"
#include "tc05.cuh"

namespace tgvkv {
namespace {

constexpr int PM = 128;                 // query rows per tile = TMEM lanes
constexpr int PN = 128;                 // keys per K / V tile
constexpr int PST = 4;                  // ring stages
constexpr int P_NSW = 4;                // softmax warps
constexpr int COPY_WARP = 2 + P_NSW;      // copies the query rows to q_text
constexpr int P_THREADS = (3 + P_NSW) * 32;
constexpr int P_TMEM_COLS = 512;        // S buffers at columns 0 and 128, O at 256
constexpr uint32_t O_COL = 256;
constexpr float kRescaleLog2 = 8.f;     // a stale reference maximum may trail by 2^8

template <int D>
struct FSmem {
    uint16_t q[2][D / 64][PM * 64];     // two Q slots; per 64 dims, 128-byte swizzled rows
    uint16_t kv[PST][D / 64][PN * 64];  // the ring, in MMA order
    uint16_t p[2][PM * 64];             // P_j: keys [64b, 64b + 64) in box b, same layout
    uint64_t full[PST], empty[PST];
    uint64_t q_full[2], q_empty[2];
    uint64_t s_full[2], s_empty[2];
    uint64_t p_full, o_done, mma_done;
    uint32_t tmem_base;
    int abort_flag, never;
    int wtile[kMaxN / PM + 1];          // first query row at or after position 128 t
};

struct PItem {
    int t, lhq, l, h, g;
};

// Item i: tile t = n_qt - 1 - i / (L H_q) (longest first), then (layer, query head).
__device__ __forceinline__ PItem prefill_item(const Problem& p, int n_qt, int i) {
    const int LHq = p.L * p.H_q;
    PItem it;
    it.t = n_qt - 1 - i / LHq;
    it.lhq = i % LHq;
    it.l = it.lhq / p.H_q;
    it.h = it.lhq % p.H_q;
    it.g = it.h / p.G;
    return it;
}

__device__ __forceinline__ bool warp_wait_all(uint64_t* bar, uint32_t parity, volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, abort);
    return __all_sync(~0u, got);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&b);
}

// O (+)= P V for one key tile: K = 128 keys in steps of 16.  P (K-major)
// advances 32 bytes inside its 128-byte rows, box b = kk / 4 holding keys
// [64b, 64b + 64); V (MN-major) advances 16 key rows = 2048 bytes.
template <int D>
__device__ __forceinline__ void pv_block(uint32_t d_tmem, uint64_t pdesc, uint32_t p_box,
                                         uint64_t vdesc, bool accumulate) {
    constexpr uint32_t IDESC_PV = tc::idesc_bf16_bmn(PM, D);
#pragma unroll
    for (int kk = 0; kk < PN / 16; ++kk) {
        const uint64_t a = pdesc + (uint64_t)((kk >> 2) * p_box + (kk & 3) * 2);
        const uint64_t b = vdesc + (uint64_t)(kk * (16 * 128 / 16));
        tc::mma_bf16(d_tmem, a, b, IDESC_PV, (accumulate || kk > 0) ? 1u : 0u);
    }
}

// Q K^T for one key tile: D / 16 MMAs of 128 x 128, K = D.
template <int D>
__device__ __forceinline__ void qk_block(uint32_t d_tmem, uint64_t qdesc, uint64_t kdesc) {
    constexpr uint32_t IDESC_QK = tc::idesc_bf16(PM, PN);
    constexpr uint32_t HALF = PM * 64 * 2 / 16;   // next 64 dims, 16-byte units
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t a = qdesc + (uint64_t)((kk >> 2) * HALF + (kk & 3) * 2);
        const uint64_t b = kdesc + (uint64_t)((kk >> 2) * HALF + (kk & 3) * 2);
        tc::mma_bf16(d_tmem, a, b, IDESC_QK, kk > 0 ? 1u : 0u);
    }
}

// One row of a score tile: P = 2^(x sl2 - m) for its 128 keys (a masked key
// holds x = -inf, so P = 0 there), packed in bf16 pairs; returns the fp32 sum.
// VISION: also adds the part over the vision keys (bits in vw, the same for
// every lane of the warp) to vs, per 32-key word: the word's sum when it is all
// vision, nothing when it is all text, key by key only for a mixed word.
template <bool VISION>
__device__ __forceinline__ float exp_row(const float (&x)[PN], float sl2, float m,
                                         const uint32_t (&vw)[4], uint32_t (&pk)[PN / 2],
                                         float& vs) {
    const float2 s2 = make_float2(sl2, sl2), n2 = make_float2(-m, -m);
    float z = 0.f;
#pragma unroll
    for (int w = 0; w < PN / 32; ++w) {
        float e[32];
        float2 za = make_float2(0.f, 0.f), zb = za;
#pragma unroll
        for (int c = 0; c < 32; c += 4) {
            const float2 t0 = fma2(make_float2(x[32 * w + c], x[32 * w + c + 1]), s2, n2);
            const float2 t1 = fma2(make_float2(x[32 * w + c + 2], x[32 * w + c + 3]), s2, n2);
            e[c] = fast_exp2(t0.x);
            e[c + 1] = fast_exp2(t0.y);
            e[c + 2] = fast_exp2(t1.x);
            e[c + 3] = fast_exp2(t1.y);
            pk[16 * w + c / 2] = pack_bf16(e[c], e[c + 1]);
            pk[16 * w + c / 2 + 1] = pack_bf16(e[c + 2], e[c + 3]);
            za = add2(za, make_float2(e[c], e[c + 1]));
            zb = add2(zb, make_float2(e[c + 2], e[c + 3]));
        }
        const float zw = (za.x + za.y) + (zb.x + zb.y);
        z += zw;
        if (VISION) {
            const uint32_t bits = vw[w];
            if (bits == ~0u) {
                vs += zw;
            } else if (bits != 0u) {
                float2 va = make_float2(0.f, 0.f);
#pragma unroll
                for (int c = 0; c < 32; c += 2)
                    va = add2(va, make_float2((bits >> c) & 1u ? e[c] : 0.f,
                                              (bits >> (c + 1)) & 1u ? e[c + 1] : 0.f));
                vs += va.x + va.y;
            }
        }
    }
    return z;
}

// Three-input maximum (PTX max.f32 with three sources).
__device__ __forceinline__ float fmax3f(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

__device__ __forceinline__ float row_max(const float (&x)[PN]) {
    float a = -INFINITY, b = -INFINITY;
#pragma unroll
    for (int c = 0; c < PN; c += 4) {
        a = fmax3f(a, x[c], x[c + 1]);
        b = fmax3f(b, x[c + 2], x[c + 3]);
    }
    return fmaxf(a, b);
}

template <int D>
__global__ void __launch_bounds__(P_THREADS, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                   const __grid_constant__ CUtensorMap tmap_v, Problem p, int n_qt, int n_items,
                   const uint16_t* __restrict__ q, const uint8_t* __restrict__ modality,
                   const int32_t* __restrict__ text_pos, uint16_t* __restrict__ o,
                   uint16_t* __restrict__ q_text, float* __restrict__ row_stats,
                   uint32_t* __restrict__ status) {
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    FSmem<D>& s = *reinterpret_cast<FSmem<D>*>(smem_raw + (((raw + 1023u) & ~1023u) - raw));
    constexpr uint32_t TILE_BYTES = (D / 64) * PN * 128;
    constexpr uint32_t BOX_UNITS = PM * 64 * 2 / 16;          // one 64-wide box, 16-byte units
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (blockIdx.x == 0) {
        for (int i = tid; i < p.n_win; i += P_THREADS) {
            const int pi = text_pos[i];
            if (pi < 0 || pi >= p.N || (i > 0 && text_pos[i - 1] >= pi))
                raise_status(status, TGVKV_STATUS_TEXT_POS);
        }
    }
    if (tid == 0) {
        s.abort_flag = 0;
        s.never = 0;
        for (int i = 0; i < PST; ++i) {
            tc::mbar_init(&s.full[i], 1);
            tc::mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&s.q_full[i], 1);
            tc::mbar_init(&s.q_empty[i], 1);
            tc::mbar_init(&s.s_full[i], 1);
            tc::mbar_init(&s.s_empty[i], P_NSW);
        }
        tc::mbar_init(&s.p_full, P_NSW);
        tc::mbar_init(&s.o_done, 1);
        tc::mbar_init(&s.mma_done, 1);
        tc::fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&s.tmem_base, P_TMEM_COLS);
        tc::tmem_relinquish();
    }
    // the query rows of each row tile t: indices wtile[t] .. wtile[t + 1] of
    // text_pos (positions ascend), as the first row at or after position 128 t
    for (int t = tid; t <= n_qt; t += P_THREADS) s.wtile[t] = p.n_win;
    __syncthreads();
    for (int i = tid; i < p.n_win; i += P_THREADS) {
        const int pi = __ldg(text_pos + i);
        if (pi >= 0 && pi < p.N) atomicMin(&s.wtile[pi / PM], i);
    }
    __syncthreads();
    if (warp == 0) {
        // suffix minimum over the tiles: per lane over a chunk, then across lanes
        const int per = (n_qt + 1 + 31) / 32;
        const int lo = lane * per, hi = lo + per < n_qt + 1 ? lo + per : n_qt + 1;
        int run = INT_MAX;
        for (int x = hi - 1; x >= lo; --x) {
            run = min(run, s.wtile[x]);
            s.wtile[x] = run;
        }
        int incl = run;                      // minimum over this lane's chunk and all later ones
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_down_sync(~0u, incl, o);
            if (lane + o < 32) incl = min(incl, y);
        }
        int later = __shfl_down_sync(~0u, incl, 1);
        if (lane == 31) later = INT_MAX;
        for (int x = lo; x < hi; ++x) s.wtile[x] = min(s.wtile[x], later);
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = s.tmem_base;
    volatile int* abort_flag = &s.abort_flag;

    // ------------------------------------------------------------ producer
    if (warp == 0 && lane == 0) {
        tc::tma_prefetch_desc(&tmap_q);
        tc::tma_prefetch_desc(&tmap_k);
        tc::tma_prefetch_desc(&tmap_v);
        int it = 0, qn[2] = {0, 0};
        bool ok = true;
        for (int i = blockIdx.x, n = 0; ok && i < n_items; i += gridDim.x, ++n) {
            const PItem itm = prefill_item(p, n_qt, i);
            const int slot = n & 1;
            if (!tc::mbar_wait(&s.q_empty[slot], ((n >> 1) & 1) ^ 1, abort_flag)) {
                ok = false;
                break;
            }
            tc::mbar_arrive_expect_tx(&s.q_full[slot], TILE_BYTES);
#pragma unroll
            for (int hd = 0; hd < D / 64; ++hd)
                tc::tma_load_2d(&s.q[slot][hd][0], &tmap_q, hd * 64, itm.lhq * p.N + itm.t * PM,
                                &s.q_full[slot]);
            ++qn[slot];
            const int kv_row = (itm.l * p.H_kv + itm.g) * p.N;
            auto load = [&](const CUtensorMap* map, int j) {
                const int stg = it % PST;
                if (!tc::mbar_wait(&s.empty[stg], ((it / PST) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    return;
                }
                tc::mbar_arrive_expect_tx(&s.full[stg], TILE_BYTES);
#pragma unroll
                for (int hd = 0; hd < D / 64; ++hd)
                    tc::tma_load_2d(&s.kv[stg][hd][0], map, hd * 64, kv_row + j * PN, &s.full[stg]);
                ++it;
            };
            const int nk = itm.t + 1;
            for (int j = 0; ok && j <= nk; ++j) {
                if (j < nk) load(&tmap_k, j);
                if (ok && j >= 1) load(&tmap_v, j - 1);
            }
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every copy this CTA issued has landed before it may exit
        for (int slot = 0; slot < 2; ++slot)
            if (qn[slot] > 0) tc::mbar_wait(&s.q_full[slot], (qn[slot] - 1) & 1, &s.never);
        for (int i = it - PST > 0 ? it - PST : 0; i < it; ++i)
            tc::mbar_wait(&s.full[i % PST], (i / PST) & 1, &s.never);
    }

    // ------------------------------------------------------------ MMA issuer
    if (warp == 1 && lane == 0) {
        const uint64_t qd0 = tc::sdesc_k_sw128(smem_u32(&s.q[0][0][0]));
        const uint64_t kd0 = tc::sdesc_k_sw128(smem_u32(&s.kv[0][0][0]));
        const uint64_t vd0 = tc::sdesc_mn_sw128(smem_u32(&s.kv[0][0][0]), PN * 64 * 2);
        const uint64_t pd0 = tc::sdesc_k_sw128(smem_u32(&s.p[0][0]));
        constexpr uint32_t Q_SLOT = (D / 64) * BOX_UNITS;
        constexpr uint32_t STAGE = (D / 64) * BOX_UNITS;
        int it = 0, st = 0, pv = 0;
        bool ok = true;
        auto qk = [&](int slot) {
            const int b = st & 1, stg = it % PST;
            bool got = tc::mbar_wait(&s.s_empty[b], ((st >> 1) & 1) ^ 1, abort_flag);
            if (got) got = tc::mbar_wait(&s.full[stg], (it / PST) & 1, abort_flag);
            if (!got) {
                ok = false;
                return;
            }
            tc::fence_after_sync();
            qk_block<D>(tmem + (uint32_t)(b * PN), qd0 + (uint64_t)(slot * Q_SLOT),
                        kd0 + (uint64_t)(stg * STAGE));
            tc::mma_commit(&s.s_full[b]);
            tc::mma_commit(&s.empty[stg]);
            ++it;
            ++st;
        };
        for (int i = blockIdx.x, n = 0; ok && i < n_items; i += gridDim.x, ++n) {
            const PItem itm = prefill_item(p, n_qt, i);
            const int slot = n & 1;
            if (!tc::mbar_wait(&s.q_full[slot], (n >> 1) & 1, abort_flag)) {
                ok = false;
                break;
            }
            const int nk = itm.t + 1;
            qk(slot);
            if (ok && nk == 1) tc::mma_commit(&s.q_empty[slot]);
            for (int j = 0; ok && j < nk; ++j) {
                if (j + 1 < nk) {
                    qk(slot);
                    if (!ok) break;
                    if (j + 2 == nk) tc::mma_commit(&s.q_empty[slot]);   // the slot's last use
                }
                // PV_j once the softmax has written P_j (and rescaled O)
                const int stg = it % PST;
                bool got = tc::mbar_wait(&s.p_full, pv & 1, abort_flag);
                if (got) got = tc::mbar_wait(&s.full[stg], (it / PST) & 1, abort_flag);
                if (!got) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                pv_block<D>(tmem + O_COL, pd0, BOX_UNITS, vd0 + (uint64_t)(stg * STAGE), j > 0);
                tc::mma_commit(&s.empty[stg]);
                tc::mma_commit(&s.o_done);
                ++it;
                ++pv;
            }
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every MMA this CTA issued has finished before TMEM is released
        tc::mma_commit(&s.mma_done);
        tc::mbar_wait(&s.mma_done, 0, &s.never);
    }

    // ------------------------------------------------------------ softmax
    if (warp >= 2 && warp < COPY_WARP) {
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;                   // this thread's row = TMEM lane
        const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
        const float sl2 = p.scale_log2;
        int st = 0, od = 0;
        bool ok = true;
        for (int i = blockIdx.x; ok && i < n_items; i += gridDim.x) {
            const PItem itm = prefill_item(p, n_qt, i);
            const int nk = itm.t + 1;
            const int pos = itm.t * PM + r;
            const bool valid = pos < p.N;
            // query row of the eviction step at this position: the tile's rows
            // are text_pos[ws .. we); those on this warp's 32 positions set bits
            const int base = itm.t * PM + quarter * 32;
            const int ws = s.wtile[itm.t], we = s.wtile[itm.t + 1];
            int wi = -1;
            if (we > ws) {
                uint32_t hit = 0u;
                int below = 0;
                for (int k0 = ws; k0 < we; k0 += 32) {
                    const int e = k0 + lane;
                    const int pe = e < we ? __ldg(text_pos + e) : INT_MAX;
                    below += __popc(__ballot_sync(~0u, pe < base));
                    const bool in = pe >= base && pe - base < 32;
                    hit |= __reduce_or_sync(~0u, in ? 1u << (pe - base) : 0u);
                }
                if (valid && ((hit >> lane) & 1u)) wi = ws + below + __popc(hit & ((1u << lane) - 1u));
            }
            const bool want_v = __any_sync(~0u, wi >= 0);
            float m = -INFINITY, lsum = 0.f, vsum = 0.f;
            // modality bytes of key tile j (this lane's keys 32 w + lane), loaded one
            // tile ahead and first used a tile later, so that the loads' latency
            // hides behind a tile of work
            int mod_next[4] = {0, 0, 0, 0};
            auto load_modality = [&](int j) {
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const int key = j * PN + 32 * w + lane;
                    mod_next[w] = key < p.N ? (int)__ldg(modality + key) : 0;
                }
            };
            if (want_v) load_modality(0);
            for (int j = 0; j < nk; ++j) {
                const int b = st & 1;
                uint32_t vw[4] = {0u, 0u, 0u, 0u};
                if (want_v) {
#pragma unroll
                    for (int w = 0; w < 4; ++w) vw[w] = __ballot_sync(~0u, mod_next[w] != 0);
                    if (j + 1 < nk) load_modality(j + 1);
                }
                if (!warp_wait_all(&s.s_full[b], (st >> 1) & 1, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                    break;
                }
                ++st;
                tc::fence_after_sync();
                float x[PN];
#pragma unroll
                for (int c = 0; c < PN / 32; ++c) {
                    float y[32];
                    tc::tmem_ld32(tl + (uint32_t)(b * PN + 32 * c), y);
#pragma unroll
                    for (int e = 0; e < 32; ++e) x[32 * c + e] = y[e];
                }
                tc::tmem_wait_ld();
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&s.s_empty[b]);

                // keys c <= r are visible in the diagonal tile, all of them below it;
                // a masked logit becomes -inf, so that 2^(x sl2 - m) is 0 there
                if (j == itm.t) {
#pragma unroll
                    for (int c = 0; c < PN; ++c)
                        if (c > r) x[c] = -INFINITY;
                }
                const float m_tile = row_max(x) * sl2;
                float alpha = 1.f;
                if (m_tile > m + kRescaleLog2) {   // also the first tile (m = -inf)
                    alpha = fast_exp2(m - m_tile);
                    m = m_tile;
                    lsum *= alpha;
                    vsum *= alpha;
                }
                uint32_t pk[PN / 2];
                // (lanes without a query row sum a vision mass that is never written)
                if (want_v)
                    lsum += exp_row<true>(x, sl2, m, vw, pk, vsum);
                else
                    lsum += exp_row<false>(x, sl2, m, vw, pk, vsum);

                // PV_{j-1} has finished: the P buffer and O are free
                if (j > 0) {
                    if (!warp_wait_all(&s.o_done, od & 1, abort_flag)) {
                        ok = false;
                        s.abort_flag = 1;
                        break;
                    }
                    ++od;
                    tc::fence_after_sync();
                    if (__any_sync(~0u, alpha != 1.f)) {
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            float y[32];
                            tc::tmem_ld32(tl + O_COL + (uint32_t)(32 * c), y);
                            tc::tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 32; ++e) y[e] *= alpha;
                            tc::tmem_st32(tl + O_COL + (uint32_t)(32 * c), y);
                        }
                        tc::tmem_wait_st();
                    }
                }
                // P row r in the 128-byte swizzled K-major layout: 16-byte chunk
                // c of box b at byte r * 128 + ((c ^ (r & 7)) << 4)
#pragma unroll
                for (int ch = 0; ch < PN / 8; ++ch) {
                    const int bx = ch >> 3, cc = ch & 7;
                    const uint32_t addr = smem_u32(&s.p[bx][0]) + (uint32_t)(r * 128 + ((cc ^ (r & 7)) << 4));
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                                 "r"(pk[4 * ch]), "r"(pk[4 * ch + 1]), "r"(pk[4 * ch + 2]),
                                 "r"(pk[4 * ch + 3])
                                 : "memory");
                }
                tc::fence_proxy_async_smem();
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&s.p_full);
            }
            if (!ok) break;

            // ---- epilogue: O / l of the finished rows, and the eviction rows' statistics
            if (!warp_wait_all(&s.o_done, od & 1, abort_flag)) {
                ok = false;
                s.abort_flag = 1;
                break;
            }
            ++od;
            tc::fence_after_sync();
            const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
            uint16_t* orow = o + ((size_t)itm.lhq * p.N + (valid ? pos : 0)) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                float y[32];
                tc::tmem_ld32(tl + O_COL + (uint32_t)(32 * c), y);
                tc::tmem_wait_ld();
                if (valid) {
#pragma unroll
                    for (int v4 = 0; v4 < 4; ++v4) {
                        uint4 u;
                        u.x = pack_bf16(y[8 * v4] * inv, y[8 * v4 + 1] * inv);
                        u.y = pack_bf16(y[8 * v4 + 2] * inv, y[8 * v4 + 3] * inv);
                        u.z = pack_bf16(y[8 * v4 + 4] * inv, y[8 * v4 + 5] * inv);
                        u.w = pack_bf16(y[8 * v4 + 6] * inv, y[8 * v4 + 7] * inv);
                        *reinterpret_cast<uint4*>(orow + 32 * c + 8 * v4) = u;
                    }
                }
            }
            tc::fence_before_sync();
            if (wi >= 0) {
                const size_t qr = ((size_t)itm.l * p.H_q + itm.h) * p.n_win + wi;
                row_stats[3 * qr] = m;
                row_stats[3 * qr + 1] = lsum;
                row_stats[3 * qr + 2] = vsum;
            }
        }
        if (!ok) raise_status(status, TGVKV_STATUS_TIMEOUT);
    }

    // ------------------------------------------------------------ query-row copies
    // q_text[l][h][r] = q[l][h][text_pos[r]], for the rows of this CTA's items,
    // D / 8 lanes per row (16 bytes each); independent of the other roles
    if (warp == COPY_WARP) {
        constexpr int LPR = D / 8, RPI = 32 / LPR;
        const int sub = lane / LPR, c = lane % LPR;
        for (int i = blockIdx.x; i < n_items; i += gridDim.x) {
            const PItem itm = prefill_item(p, n_qt, i);
            const int ws = s.wtile[itm.t], we = s.wtile[itm.t + 1];
            const size_t qrow = ((size_t)itm.l * p.H_q + itm.h) * p.n_win;
#pragma unroll 4
            for (int e = ws + sub; e < we; e += RPI) {
                const int pos = __ldg(text_pos + e);
                if (pos < 0 || pos >= p.N) continue;
                const uint4 v4 = __ldg(reinterpret_cast<const uint4*>(q + ((size_t)itm.lhq * p.N + pos) * D) + c);
                reinterpret_cast<uint4*>(q_text + (qrow + e) * D)[c] = v4;
            }
        }
    }

    // ------------------------------------------------------------ teardown
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, P_TMEM_COLS);
    }
}

template <int D>
cudaError_t launch_prefill_d(const Problem& p, const uint16_t* q, const uint16_t* k,
                             const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                             uint16_t* o, uint16_t* q_text, float* row_stats, uint32_t* status,
                             cudaStream_t stream) {
    static_assert(sizeof(FSmem<D>) + 1024 <= 227 * 1024, "shared memory of one CTA");
    alignas(64) CUtensorMap mq, mk, mv;
    if (!make_tile_map(&mq, q, (uint64_t)p.L * p.H_q * p.N, D, PM) ||
        !make_tile_map(&mk, k, (uint64_t)p.L * p.H_kv * p.N, D, PN) ||
        !make_tile_map(&mv, v, (uint64_t)p.L * p.H_kv * p.N, D, PN))
        return cudaErrorInvalidValue;
    const size_t smem = sizeof(FSmem<D>) + 1024;
    cudaError_t e = cudaFuncSetAttribute(prefill_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    const int sms = device_sm_count();
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int n_qt = (p.N + PM - 1) / PM;
    const int n_items = p.L * p.H_q * n_qt;
    const int grid = n_items < sms ? n_items : sms;
    prefill_kernel<D><<<grid, P_THREADS, smem, stream>>>(mq, mk, mv, p, n_qt, n_items, q, modality,
                                                         text_pos, o, q_text, row_stats, status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefill(const Problem& p, const uint16_t* q, const uint16_t* k,
                           const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                           uint16_t* o, uint16_t* q_text, float* row_stats, uint32_t* status,
                           cudaStream_t stream) {
    if (p.d == 64)
        return launch_prefill_d<64>(p, q, k, v, modality, text_pos, o, q_text, row_stats, status,
                                    stream);
    return launch_prefill_d<128>(p, q, k, v, modality, text_pos, o, q_text, row_stats, status,
                                 stream);
}

}  // namespace tgvkv
