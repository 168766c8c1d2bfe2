// TWR scores and TVB statistic on the 5th-generation tensor cores (tcgen05):
// a persistent, warp-specialised kernel with one CTA per SM.
//
// The query rows of one (layer, KV head) -- the G query heads of the group
// stacked over the n_win text-query rows -- are cut into 128-row tiles.  Each
// row tile streams the head's 128-key tiles twice, the two passes of
// Eq. 2 / Eq. 8:
//
//   pass A  S = Q K^T  (TMEM lane = query row): per row an online maximum m_i,
//           normaliser Z_i and vision mass V_i over every visible key (causal:
//           key j <= position of row i).
//   pass B  S^T = K Q^T  (TMEM lane = key) over the tiles that hold vision
//           keys: per key j the sum over rows of c_i 2^(x_ij - m_i),
//           c_i = w_i / (G Z_i) -- the text-weighted column sum of Eq. 8 with
//           the GQA mean folded in.  c_i goes into the exponent,
//           2^(x_ij - m'_i) with m'_i = m_i - log2 c_i, so a term is one
//           packed-pair FFMA, one EX2 and one packed FADD, and the column sum
//           needs no cross-lane reduction.
//
// Delivering K tiles is what bounds this kernel, so every K tile loaded is
// used for as many query rows as possible: a work item is a PAIR of row tiles
// of one head (when the head has more than one), and each K tile feeds two
// MMAs, one per row tile.  A head with a single row tile is one item.
//
// Roles: warp 0 fetches items from a global counter (longest items first) and
// issues TMA loads -- the item's Q tiles, then every K tile of both passes
// through a 4-stage ring, running ahead into the next item; warp 1 owns the
// SM's 512 TMEM columns (two 128-column fp32 accumulators per softmax group)
// and one of its lanes issues the MMAs; warps 2-17 form two softmax groups.
// With a row-tile pair, group g owns row tile g; with a single row tile the
// groups take alternate K tiles.  In a group, two warps per TMEM lane quarter
// split a tile's 128 columns.  Every wait is bounded (1 s); a timeout sets
// TGVKV_STATUS_TIMEOUT and the CTA unwinds.
//
// Query rows are spread evenly over the four lane quarters (row q*rpg + i ->
// lane 32q + i) so that all softmax warps share the work when a row tile has
// fewer than 128 rows.  Row tiles of a head write partial score rows; the last
// one to finish adds them in tile order, and the last head of a layer adds the
// TV masses in head order, so the results do not depend on the schedule.
#include <cudaTypedefs.h>
#include <limits.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "launch.h"
#include "tc05.cuh"

namespace tgvkv {
namespace {

constexpr int BM = 128;           // query rows per row tile = TMEM lanes
constexpr int BN = 128;           // keys per tile
constexpr int STAGES = 4;         // K tiles in flight
constexpr int NGRP = 2;           // softmax groups
constexpr int NQB = 2;            // Q tiles in shared memory
constexpr int NIQ = 2;            // items fetched ahead
constexpr int GSOFT = 256;        // threads per softmax group (2 warps per lane quarter)
constexpr int NSOFT = NGRP * GSOFT;
constexpr int MMA2_WARP = 2 + NSOFT / 32;   // the second MMA issuer, after the softmax warps
constexpr int NTHREADS = 64 + NSOFT + 32;
constexpr int TMEM_COLS = 512;    // 2 accumulators x 2 groups x 128 columns
constexpr int MAXT = kMaxN / BN;  // key tiles per head
constexpr int MAX_RT = 256;       // row tiles per KV head (G * n_win <= 32768)
constexpr uint32_t IDESC = tc::idesc_bf16(128, 128);

template <int D>
struct PSmem {
    uint16_t q[NQB][D / 64][BM * 64];        // Q tiles, one 128-byte-swizzled half per 64 dims
    uint16_t k[STAGES][D / 64][BN * 64];     // K ring
    uint64_t full[STAGES], empty[STAGES];
    uint64_t s_full[NGRP][2], s_empty[NGRP][2];
    uint64_t q_full[NQB], q_empty[NQB], mma_done;
    uint64_t it_full[NIQ], it_empty[NIQ];
    uint64_t pb_full[NGRP][4][2], pb_empty[NGRP][4][2];  // pass-B hand-off per group and quarter
    uint32_t vmask[MAXT][4];                 // vision bit of each key of each tile
    int vis_before[MAXT + 1];                // vision keys before each tile
    int rt_max[MAX_RT], rt_min[MAX_RT];      // per row tile: max / min query position
    alignas(16) int row_pos[NGRP][BM];       // per group and TMEM lane: row position, -1 = none
    alignas(16) float row_nmp[NGRP][BM];     // -(m_i - log2 c_i); -inf = no row
    float row_w[NGRP][BM], row_mass[NGRP][BM];
    float part_m[NGRP * 2][BM], part_z[NGRP * 2][BM], part_v[NGRP * 2][BM];
    float pbuf[NGRP][2][BM];
    int item_q[NIQ];
    uint32_t tmem_base;
    int abort_flag, never, stop, head_last, cur_item;
    int issued[NGRP];                        // accumulator uses issued so far, per group
    float tile_mass[NGRP];
};

// One work item: one or two row tiles of one (layer, KV head).
struct Item {
    int lh, l, g, nr, ntmax;
    int t[2], nt[2], rows[2], rpg[2], minp[2];
    // element r (0 or 1) without a run-time array index
    __device__ __forceinline__ static int pick(const int (&a)[2], int r) { return r ? a[1] : a[0]; }
};

template <int D>
__device__ __forceinline__ Item item_info(const Problem& p, const PSmem<D>& s, int id, int npair,
                                          bool pair) {
    Item it;
    it.lh = id / npair;
    const int tp = npair - 1 - id % npair;   // later row tiles (longer causal range) first
    it.l = it.lh / p.H_kv;
    it.g = it.lh % p.H_kv;
    it.t[0] = pair ? 2 * tp : tp;
    it.t[1] = (pair && 2 * tp + 1 < p.T) ? 2 * tp + 1 : -1;
    it.nr = it.t[1] >= 0 ? 2 : 1;
    it.ntmax = 0;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int t = it.t[r] >= 0 ? it.t[r] : it.t[0];
        it.rows[r] = min(BM, p.R - t * BM);
        it.rpg[r] = (it.rows[r] + 3) >> 2;
        it.nt[r] = (s.rt_max[t] + BN) / BN;
        it.minp[r] = s.rt_min[t];
    }
    it.ntmax = it.nr == 2 ? max(it.nt[0], it.nt[1]) : it.nt[0];
    return it;
}

// One 128 x 128 x D product into the accumulator at d_tmem: D/16 MMAs whose
// operand descriptors differ from the tile's base descriptors by constants
// (K offset of 32 bytes inside a 128-byte swizzle atom, 16 KB per 64 dims).
// Pass A: S = Q K^T (TRANS = false); pass B: S^T = K Q^T.
template <int D, bool TRANS>
__device__ __forceinline__ void mma_kq(uint32_t d_tmem, uint64_t qd, uint64_t kd) {
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t o = (uint64_t)((kk >> 2) * (BM * 64 * 2 / 16) + (kk & 3) * 2);
        const uint64_t a = TRANS ? kd + o : qd + o, b = TRANS ? qd + o : kd + o;
        if (kk == 0)
            tc::mma_bf16_c<0>(d_tmem, a, b, IDESC);
        else
            tc::mma_bf16_c<1>(d_tmem, a, b, IDESC);
    }
}

__device__ __forceinline__ int next_vis_tile(const int* vis_before, int kt, int n_tiles) {
    while (kt < n_tiles && vis_before[kt + 1] == vis_before[kt]) ++kt;
    return kt;
}

__device__ __forceinline__ float max32(const float (&x)[32]) {
    float a = fmaxf(x[0], x[1]), b = fmaxf(x[2], x[3]), c = fmaxf(x[4], x[5]), d = fmaxf(x[6], x[7]);
#pragma unroll
    for (int i = 8; i < 32; i += 4) {
        a = fmaxf(a, x[i]);
        b = fmaxf(b, x[i + 1]);
        c = fmaxf(c, x[i + 2]);
        d = fmaxf(d, x[i + 3]);
    }
    return fmaxf(fmaxf(a, b), fmaxf(c, d));
}

__device__ __forceinline__ float max32_masked(const float (&x)[32], int lim) {
    float a = -INFINITY, b = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
        if (i <= lim) a = fmaxf(a, x[i]);
        if (i + 1 <= lim) b = fmaxf(b, x[i + 1]);
    }
    return fmaxf(a, b);
}

// Sum of e_c = 2^(x_c sl2 + nm) over one 32-key word (columns c <= lim when
// MASKED), and the part of it over the vision keys flagged in vm.  Exponent
// arguments and sums run on packed fp32 pairs.
template <bool MASKED>
__device__ __forceinline__ void exp_word(const float (&x)[32], float sl2, float nm, int lim,
                                         uint32_t vm, float& z, float& v) {
    const float2 s2 = make_float2(sl2, sl2), n2 = make_float2(nm, nm);
    float2 za = make_float2(0.f, 0.f), zb = za;
    if (vm == 0u || vm == 0xFFFFFFFFu) {
#pragma unroll
        for (int c = 0; c < 32; c += 4) {
            const float2 t0 = fma2(make_float2(x[c], x[c + 1]), s2, n2);
            const float2 t1 = fma2(make_float2(x[c + 2], x[c + 3]), s2, n2);
            float2 e0 = make_float2(fast_exp2(t0.x), fast_exp2(t0.y));
            float2 e1 = make_float2(fast_exp2(t1.x), fast_exp2(t1.y));
            if (MASKED) {
                if (c > lim) e0.x = 0.f;
                if (c + 1 > lim) e0.y = 0.f;
                if (c + 2 > lim) e1.x = 0.f;
                if (c + 3 > lim) e1.y = 0.f;
            }
            za = add2(za, e0);
            zb = add2(zb, e1);
        }
        const float zs = (za.x + za.y) + (zb.x + zb.y);
        z += zs;
        if (vm) v += zs;
    } else {
        float2 va = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
            const float2 t = fma2(make_float2(x[c], x[c + 1]), s2, n2);
            float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
            if (MASKED) {
                if (c > lim) e.x = 0.f;
                if (c + 1 > lim) e.y = 0.f;
            }
            za = add2(za, e);
            va = add2(va, make_float2((vm >> c) & 1u ? e.x : 0.f, (vm >> (c + 1)) & 1u ? e.y : 0.f));
        }
        z += za.x + za.y;
        v += va.x + va.y;
    }
}

// Sum over the valid rows of one 32-row group of 2^(y_i sl2 + nmp_i), with the
// causal mask j <= pos_i unless every row sees key j.  FULL: all 32 rows exist.
template <bool FULL>
__device__ __forceinline__ float colsum_group(const float (&y)[32], const float* nmp,
                                              const int* pos, float sl2, int rpg, int j,
                                              bool all_vis) {
    const float2 s2 = make_float2(sl2, sl2);
    float2 a = make_float2(0.f, 0.f), b = a;
#pragma unroll
    for (int i = 0; i < 32; i += 4) {
        if (FULL || i < rpg) {
            const float4 n4 = *reinterpret_cast<const float4*>(nmp + i);
            const float2 t0 = fma2(make_float2(y[i], y[i + 1]), s2, make_float2(n4.x, n4.y));
            const float2 t1 = fma2(make_float2(y[i + 2], y[i + 3]), s2, make_float2(n4.z, n4.w));
            float2 e0 = make_float2(fast_exp2(t0.x), fast_exp2(t0.y));
            float2 e1 = make_float2(fast_exp2(t1.x), fast_exp2(t1.y));
            if (!all_vis) {
                const int4 p4 = *reinterpret_cast<const int4*>(pos + i);
                if (j > p4.x) e0.x = 0.f;
                if (j > p4.y) e0.y = 0.f;
                if (j > p4.z) e1.x = 0.f;
                if (j > p4.w) e1.y = 0.f;
            }
            a = add2(a, e0);
            b = add2(b, e1);
        }
    }
    return (a.x + a.y) + (b.x + b.y);
}

// Bounded wait until *counter == value (the other MMA issuer has issued the
// group's previous accumulator use).
__device__ __forceinline__ bool wait_turn(const int* counter, int value, volatile int* abort) {
    const volatile int* c = counter;
    if (*c == value) return true;
    const long long c0 = clock64();
    for (uint32_t i = 1;; ++i) {
        if (*c == value) return true;
        if ((i & 63u) == 0) {
            if (*abort) return false;
            if (clock64() - c0 > tc::kWaitLimitCycles) return false;
        }
    }
}

// A bounded wait whose outcome is the same for every lane of the warp (the
// tensor-memory loads that follow are warp-collective).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, abort);
    return __all_sync(~0u, got);
}

template <int D>
__global__ void __launch_bounds__(NTHREADS, 1)
score_tc_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                Problem p, const uint8_t* __restrict__ modality,
                const int32_t* __restrict__ text_pos, const float* __restrict__ w,
                float* __restrict__ scores, float* __restrict__ tvb_stat,
                float* __restrict__ score_part, float* __restrict__ stat_part,
                float* __restrict__ stat_head, uint32_t* __restrict__ tickets,
                uint32_t* __restrict__ status) {
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    PSmem<D>& s = *reinterpret_cast<PSmem<D>*>(smem_raw + (((raw + 1023u) & ~1023u) - raw));
    constexpr uint32_t TILE_BYTES = (D / 64) * BN * 128;   // one K tile = one Q tile

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int T = p.T;
    const bool pair = T >= 2;
    const int npair = pair ? (T + 1) / 2 : 1;
    const int n_items = p.L * p.H_kv * npair;
    const float sl2 = p.scale_log2;
    uint32_t* work_counter = tickets + p.L * p.H_kv + p.L;
    uint32_t* done_counter = work_counter + 1;

    // ------------------------------------------------------------ prologue
    if (blockIdx.x == 0) {
        for (int i = tid; i < p.n_win; i += NTHREADS) {
            const int pi = text_pos[i];
            if (pi < 0 || pi >= p.N || (i > 0 && text_pos[i - 1] >= pi))
                raise_status(status, TGVKV_STATUS_TEXT_POS);
        }
    }
    if (tid == 0) {
        s.abort_flag = 0;
        s.never = 0;
        for (int gp = 0; gp < NGRP; ++gp) s.issued[gp] = 0;
        for (int i = 0; i < STAGES; ++i) {
            tc::mbar_init(&s.full[i], 1);
            tc::mbar_init(&s.empty[i], 1);
        }
        for (int gp = 0; gp < NGRP; ++gp)
            for (int i = 0; i < 2; ++i) {
                tc::mbar_init(&s.s_full[gp][i], 1);
                tc::mbar_init(&s.s_empty[gp][i], GSOFT / 32);   // one arrival per warp of the group
            }
        for (int i = 0; i < NQB; ++i) {
            tc::mbar_init(&s.q_full[i], 1);
            tc::mbar_init(&s.q_empty[i], 2);    // both MMA issuers
        }
        for (int i = 0; i < NIQ; ++i) {
            tc::mbar_init(&s.it_full[i], 1);
            tc::mbar_init(&s.it_empty[i], 3);   // the two MMA issuers and the softmax role
        }
        for (int gp = 0; gp < NGRP; ++gp)
            for (int qq = 0; qq < 4; ++qq)
                for (int i = 0; i < 2; ++i) {
                    tc::mbar_init(&s.pb_full[gp][qq][i], 1);   // the writer warp of the quarter
                    tc::mbar_init(&s.pb_empty[gp][qq][i], 1);  // the reader warp
                }
        tc::mbar_init(&s.mma_done, 2);
        tc::fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&s.tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    const int n_tiles_all = (p.N + BN - 1) / BN;
    for (int kt = warp; kt < n_tiles_all; kt += NTHREADS / 32) {
        int cnt = 0;
#pragma unroll
        for (int wd = 0; wd < 4; ++wd) {
            const int j = kt * BN + wd * 32 + lane;
            const unsigned m = __ballot_sync(~0u, j < p.N && modality[j] != 0);
            if (lane == 0) s.vmask[kt][wd] = m;
            cnt += __popc(m);
        }
        if (lane == 0) s.vis_before[kt] = cnt;
    }
    for (int t = tid; t < T; t += NTHREADS) {
        s.rt_max[t] = -1;
        s.rt_min[t] = INT_MAX;
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    for (int r = tid; r < p.R; r += NTHREADS) {
        const int pos = text_pos[r % p.n_win];
        if (pos >= 0 && pos < p.N) {
            atomicMax(&s.rt_max[r / BM], pos);
            atomicMin(&s.rt_min[r / BM], pos);
        }
    }
    if (warp == 0) {
        const int per = (n_tiles_all + 31) / 32;
        const int b = lane * per, e = min(b + per, n_tiles_all);
        int sum = 0;
        for (int x = b; x < e; ++x) sum += s.vis_before[x];
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(~0u, incl, o);
            if (lane >= o) incl += y;
        }
        int run = incl - sum;
        for (int x = b; x < e; ++x) {
            const int c = s.vis_before[x];
            s.vis_before[x] = run;
            run += c;
        }
        const int total = __shfl_sync(~0u, incl, 31);
        if (lane == 0) {
            s.vis_before[n_tiles_all] = total;
            if (blockIdx.x == 0 && total != p.N_v) raise_status(status, TGVKV_STATUS_VISION_COUNT);
        }
    }
    __syncthreads();
    const uint32_t tmem = s.tmem_base;
    volatile int* abort_flag = &s.abort_flag;

    // ------------------------------------------------------------ producer
    if (warp == 0 && lane == 0) {
        tc::tma_prefetch_desc(&tmap_q);
        tc::tma_prefetch_desc(&tmap_k);
        int it = 0, qn = 0;
        bool ok = true;
        for (int n = 0; ok; ++n) {
            // fetch the next item (or the end mark) for every role of this CTA
            const int slot = n % NIQ;
            if (!tc::mbar_wait(&s.it_empty[slot], ((n / NIQ) & 1) ^ 1, abort_flag)) {
                ok = false;
                break;
            }
            const int id = (int)atomicAdd(work_counter, 1u);
            s.item_q[slot] = id < n_items ? id : -1;
            tc::mbar_arrive(&s.it_full[slot]);
            if (id >= n_items) {
                // the last CTA to run out of work re-arms the counters for the next launch
                if (atomicAdd(done_counter, 1u) == gridDim.x - 1) {
                    *work_counter = 0u;
                    *done_counter = 0u;
                }
                break;
            }
            const Item itm = item_info(p, s, id, npair, pair);
            for (int r = 0; r < itm.nr; ++r, ++qn) {
                const int qb = qn % NQB;
                if (!tc::mbar_wait(&s.q_empty[qb], ((qn / NQB) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const int qy = (itm.l * p.H_q + itm.g * p.G) * p.n_win + Item::pick(itm.t, r) * BM;
                tc::mbar_arrive_expect_tx(&s.q_full[qb], TILE_BYTES);
#pragma unroll
                for (int qg = 0; qg < 4; ++qg)
#pragma unroll
                    for (int h = 0; h < D / 64; ++h)
                        tc::tma_load_2d(&s.q[qb][h][qg * 32 * 64], &tmap_q, h * 64,
                                        qy + qg * Item::pick(itm.rpg, r), &s.q_full[qb]);
            }
            auto issue = [&](int kt) {
                const int stage = it % STAGES;
                if (!tc::mbar_wait(&s.empty[stage], ((it / STAGES) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    return;
                }
                tc::mbar_arrive_expect_tx(&s.full[stage], TILE_BYTES);
#pragma unroll
                for (int h = 0; h < D / 64; ++h)
                    tc::tma_load_2d(&s.k[stage][h][0], &tmap_k, h * 64, itm.lh * p.N + kt * BN,
                                    &s.full[stage]);
                ++it;
            };
            for (int kt = 0; ok && kt < itm.ntmax; ++kt) issue(kt);
            for (int kt = next_vis_tile(s.vis_before, 0, itm.ntmax); ok && kt < itm.ntmax;
                 kt = next_vis_tile(s.vis_before, kt + 1, itm.ntmax))
                issue(kt);
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every copy this CTA issued has landed before it may exit
        for (int i = max(0, qn - NQB); i < qn; ++i)
            tc::mbar_wait(&s.q_full[i % NQB], (i / NQB) & 1, &s.never);
        for (int i = max(0, it - STAGES); i < it; ++i)
            tc::mbar_wait(&s.full[i % STAGES], (i / STAGES) & 1, &s.never);
    }

    // ------------------------------------------------------------ MMA issuers
    // Two threads in different warps issue the MMAs of alternate ring entries.
    // A thread that uses the outcome of an mbarrier wait stalls until its own
    // MMAs in flight have drained; with two issuers the other one keeps the
    // tensor pipe busy meanwhile.  Both walk every entry to keep the
    // accumulator counters, and issue only for entries of their parity.
    // A group's accumulator uses are issued strictly in order across the two
    // threads (s.issued): when a group skips an entry, the buffer a thread
    // fills changes, and without the ordering one thread could wait on the
    // release of use u-2 before the other has issued it -- two phases behind,
    // which a parity wait cannot tell apart from a completed phase.
    if ((warp == 1 || warp == MMA2_WARP) && lane == 0) {
        const int me = warp == 1 ? 0 : 1;
        // shared-memory descriptors, computed once: the start-address field
        // (16-byte units, < 2^14 inside 256 KB) takes plain additions
        const uint64_t kdesc0 = tc::sdesc_k_sw128(smem_u32(&s.k[0][0][0]));
        const uint64_t qdesc0 = tc::sdesc_k_sw128(smem_u32(&s.q[0][0][0]));
        constexpr uint32_t KSTAGE_DESC = (uint32_t)(sizeof(s.k[0]) >> 4);
        constexpr uint32_t QBUF_DESC = (uint32_t)(sizeof(s.q[0]) >> 4);
        int it = 0, qn = 0;
        int acc[NGRP] = {0, 0};
        bool ok = true;
        for (int n = 0; ok; ++n) {
            const int slot = n % NIQ;
            if (!tc::mbar_wait(&s.it_full[slot], (n / NIQ) & 1, abort_flag)) {
                ok = false;
                break;
            }
            const int id = s.item_q[slot];
            tc::mbar_arrive(&s.it_empty[slot]);
            if (id < 0) break;
            const Item itm = item_info(p, s, id, npair, pair);
            // Q tiles of this item: slot qb0 (and qb1 for a pair)
            const int qb0 = qn % NQB, qb1 = (qn + 1) % NQB;
            for (int r = 0; r < itm.nr; ++r, ++qn) {
                if (!tc::mbar_wait(&s.q_full[qn % NQB], (qn / NQB) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
            }
            if (!ok) break;
            // descriptors of the item's Q tiles; a K stage's is kdesc0 + stage * KSTAGE_DESC
            const uint64_t qd0 = qdesc0 + (uint64_t)(qb0 * QBUF_DESC);
            const uint64_t qd1 = qdesc0 + (uint64_t)(qb1 * QBUF_DESC);
            int local = 0;
            auto mma_tile = [&](int kt, bool transposed) {
                const int stage = it % STAGES;
                const bool issue = (it & 1) == me;
                if (issue && !tc::mbar_wait(&s.full[stage], (it / STAGES) & 1, abort_flag)) {
                    ok = false;
                    return;
                }
                const uint64_t kd = kdesc0 + (uint64_t)(stage * KSTAGE_DESC);
#pragma unroll
                for (int gp = 0; gp < NGRP; ++gp) {
                    // which group receives an accumulator for this tile, and from which Q tile
                    const bool mine = itm.nr == 2 ? kt < itm.nt[gp] : (local & 1) == gp;
                    if (!mine) continue;
                    const int b = acc[gp] & 1;
                    if (!issue) {
                        ++acc[gp];
                        continue;
                    }
                    if (!wait_turn(&s.issued[gp], acc[gp], abort_flag) ||
                        !tc::mbar_wait(&s.s_empty[gp][b], ((acc[gp] >> 1) & 1) ^ 1, abort_flag)) {
                        ok = false;
                        return;
                    }
                    tc::fence_after_sync();
                    const uint32_t d_tmem = tmem + (uint32_t)((gp * 2 + b) * BN);
                    const uint64_t qd = (itm.nr == 2 && gp == 1) ? qd1 : qd0;
                    if (transposed)
                        mma_kq<D, true>(d_tmem, qd, kd);
                    else
                        mma_kq<D, false>(d_tmem, qd, kd);
                    tc::mma_commit(&s.s_full[gp][b]);
                    ++acc[gp];
                    *reinterpret_cast<volatile int*>(&s.issued[gp]) = acc[gp];
                }
                if (issue) tc::mma_commit(&s.empty[stage]);
                ++it;
                ++local;
            };
            for (int kt = 0; ok && kt < itm.ntmax; ++kt) mma_tile(kt, false);
            for (int kt = next_vis_tile(s.vis_before, 0, itm.ntmax); ok && kt < itm.ntmax;
                 kt = next_vis_tile(s.vis_before, kt + 1, itm.ntmax))
                mma_tile(kt, true);
            // the item's Q tiles are free once these MMAs finish
            tc::mma_commit(&s.q_empty[qb0]);
            if (itm.nr == 2) tc::mma_commit(&s.q_empty[qb1]);
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every MMA this CTA issued has finished before TMEM is released
        tc::mma_commit(&s.mma_done);
        tc::mbar_wait(&s.mma_done, 0, &s.never);
    }

    // ------------------------------------------------------------ softmax groups
    if (warp >= 2 && warp < MMA2_WARP) {
        const int sid = tid - 64;
        const int quarter = warp & 3;
        const int grp = (warp - 2) >> 3;
        const int wq = ((warp - 2) >> 2) & 1;               // which 64 columns of a tile
        const int ln = quarter * 32 + lane;                 // this thread's TMEM lane
        const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(wq * 64);
        int acc_n = 0, u = 0;
        bool ok = true;
        for (int n = 0;; ++n) {
            // ---- the item, as fetched by the producer
            const int slot = n % NIQ;
            if (sid == 0) {
                const bool got = tc::mbar_wait(&s.it_full[slot], (n / NIQ) & 1, abort_flag);
                s.cur_item = got ? s.item_q[slot] : -1;
                if (!got) {
                    s.abort_flag = 1;
                    ok = false;
                } else {
                    tc::mbar_arrive(&s.it_empty[slot]);
                }
            }
            tc::named_bar_sync(1, NSOFT);
            const int id = s.cur_item;
            if (id < 0) break;
            const Item itm = item_info(p, s, id, npair, pair);
            const int r = itm.nr == 2 ? grp : 0;          // this group's row tile
            const int t = Item::pick(itm.t, r);
            const int rows_t = Item::pick(itm.rows, r), rpg = Item::pick(itm.rpg, r);
            const int n_mine = itm.nr == 2 ? Item::pick(itm.nt, r) : itm.ntmax;   // tiles with this group's rows
            const int min_pos = Item::pick(itm.minp, r);
            float* out = (T == 1) ? scores + (size_t)itm.lh * p.N_v
                                  : score_part + ((size_t)itm.lh * T + t) * p.N_v;

            // ---- rows of this group's row tile: lane 32q + i holds row q*rpg + i
            if (wq == 0) {
                const int rr = quarter * rpg + lane;
                int pos = -1;
                float wr = 0.f;
                if (lane < rpg && rr < rows_t) {
                    const int wi = (t * BM + rr) % p.n_win;
                    pos = text_pos[wi];
                    if (pos < 0 || pos >= p.N) pos = -1;
                    wr = w[(long long)itm.l * p.w_stride + wi];
                    if (!(wr >= 0.f) || isinf(wr)) {
                        raise_status(status, TGVKV_STATUS_WEIGHT);
                        wr = 0.f;
                    }
                }
                s.row_pos[grp][ln] = pos;
                s.row_w[grp][ln] = wr;
            }
            tc::named_bar_sync(1, NSOFT);
            const int my_pos = s.row_pos[grp][ln];

            // ---- pass A: statistics of this thread's row over its 64 columns of its tiles
            float m = -INFINITY, z = 0.f, v = 0.f;
            int local = 0;
            for (int kt = 0; ok && kt < itm.ntmax; ++kt, ++local) {
                const bool mine = itm.nr == 2 ? kt < n_mine : (local & 1) == grp;
                if (!mine) continue;
                const int b = acc_n & 1;
                if (!warp_wait(&s.s_full[grp][b], (acc_n >> 1) & 1, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                    break;
                }
                tc::fence_after_sync();
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float x[32];
                    tc::tmem_ld32(tl + (uint32_t)((grp * 2 + b) * BN + h * 32), x);
                    tc::tmem_wait_ld();
                    if (h == 1) {
                        tc::fence_before_sync();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(&s.s_empty[grp][b]);
                    }
                    const int lim = my_pos - (kt * BN + wq * 64 + h * 32);   // columns 0..lim visible
                    if (lim >= 0) {
                        const uint32_t vm = s.vmask[kt][wq * 2 + h];
                        if (lim >= 31) {
                            const float m_new = fmaxf(m, max32(x) * sl2);
                            const float alpha = fast_exp2(m - m_new);
                            z *= alpha;
                            v *= alpha;
                            exp_word<false>(x, sl2, -m_new, 31, vm, z, v);
                            m = m_new;
                        } else {
                            const float m_new = fmaxf(m, max32_masked(x, lim) * sl2);
                            const float alpha = fast_exp2(m - m_new);
                            z *= alpha;
                            v *= alpha;
                            exp_word<true>(x, sl2, -m_new, lim, vm, z, v);
                            m = m_new;
                        }
                    }
                }
                ++acc_n;
            }
            // ---- combine the partial statistics of each row
            s.part_m[grp * 2 + wq][ln] = m;
            s.part_z[grp * 2 + wq][ln] = z;
            s.part_v[grp * 2 + wq][ln] = v;
            tc::named_bar_sync(1, NSOFT);
            if (wq == 0) {
                // one row tile: all four parts; two: this group's two
                const int c0 = itm.nr == 2 ? grp * 2 : 0, c1 = itm.nr == 2 ? grp * 2 + 2 : 4;
                float mt = -INFINITY;
                for (int c = c0; c < c1; ++c) mt = fmaxf(mt, s.part_m[c][ln]);
                float zt = 0.f, vt = 0.f;
                if (mt != -INFINITY) {
                    for (int c = c0; c < c1; ++c) {
                        const float a = fast_exp2(s.part_m[c][ln] - mt);
                        zt += s.part_z[c][ln] * a;
                        vt += s.part_v[c][ln] * a;
                    }
                }
                const bool valid = my_pos >= 0 && zt > 0.f;
                // rows without attention get -m' = -inf: every term 2^-inf = 0
                s.row_nmp[grp][ln] =
                    valid ? fast_log2(s.row_w[grp][ln] / ((float)p.G * zt)) - mt : -INFINITY;
                s.row_mass[grp][ln] = valid ? vt / zt : 0.f;
            }
            tc::named_bar_sync(1, NSOFT);
            if (wq == 0 && quarter == 0) {
                // TV mass of this group's row tile, in lane order
                float a = (s.row_mass[grp][lane] + s.row_mass[grp][lane + 32]) +
                          (s.row_mass[grp][lane + 64] + s.row_mass[grp][lane + 96]);
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(~0u, a, o);
                if (lane == 0) s.tile_mass[grp] = a;
            }

            // ---- pass B: text-weighted column sums, one key per thread
            const float* nmp = s.row_nmp[grp] + wq * 64;
            const int* rp = s.row_pos[grp] + wq * 64;
            const bool full_groups = rpg == 32;
            for (int kt = next_vis_tile(s.vis_before, 0, itm.ntmax); ok && kt < itm.ntmax;
                 kt = next_vis_tile(s.vis_before, kt + 1, itm.ntmax), ++local) {
                const bool mine = itm.nr == 2 ? kt < n_mine : (local & 1) == grp;
                if (!mine) continue;
                const int b = acc_n & 1;
                if (!warp_wait(&s.s_full[grp][b], (acc_n >> 1) & 1, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                    break;
                }
                tc::fence_after_sync();
                const int j = kt * BN + ln;                     // this thread's key
                const bool all_vis = kt * BN + BN - 1 <= min_pos;
                float sum = 0.f;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float y[32];
                    tc::tmem_ld32(tl + (uint32_t)((grp * 2 + b) * BN + h * 32), y);
                    tc::tmem_wait_ld();
                    if (h == 1) {
                        tc::fence_before_sync();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(&s.s_empty[grp][b]);
                    }
                    if (full_groups)
                        sum += colsum_group<true>(y, nmp + h * 32, rp + h * 32, sl2, rpg, j, all_vis);
                    else
                        sum += colsum_group<false>(y, nmp + h * 32, rp + h * 32, sl2, rpg, j, all_vis);
                }
                ++acc_n;
                // the two column halves of key j meet at the wq == 0 warp of the group
                const int b2 = u & 1;
                const uint32_t ph = (u >> 1) & 1;
                ++u;
                if (wq == 1) {
                    if (!warp_wait(&s.pb_empty[grp][quarter][b2], ph ^ 1, abort_flag)) {
                        ok = false;
                        s.abort_flag = 1;
                        break;
                    }
                    s.pbuf[grp][b2][ln] = sum;
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&s.pb_full[grp][quarter][b2]);
                } else {
                    if (!warp_wait(&s.pb_full[grp][quarter][b2], ph, abort_flag)) {
                        ok = false;
                        s.abort_flag = 1;
                        break;
                    }
                    sum += s.pbuf[grp][b2][ln];
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&s.pb_empty[grp][quarter][b2]);
                    const uint32_t word = s.vmask[kt][quarter];
                    if (j < p.N && ((word >> lane) & 1u)) {
                        int vr = s.vis_before[kt] + __popc(word & ((1u << lane) - 1u));
                        for (int q2 = 0; q2 < quarter; ++q2) vr += __popc(s.vmask[kt][q2]);
                        if (vr < p.N_v) out[vr] = sum;
                    }
                }
            }
            // vision keys after every query row of this row tile get no attention
            if (itm.nr == 2 || grp == 0)
                for (int vv = s.vis_before[n_mine] + (sid & (GSOFT - 1)); vv < p.N_v; vv += GSOFT)
                    out[vv] = 0.f;

            // ---- reductions over row tiles (per head) and heads (per layer)
            __threadfence();
            if (sid == 0) s.stop = *abort_flag;
            tc::named_bar_sync(1, NSOFT);
            if (sid == 0) {
                int last = 0;
                if (T == 1) {
                    stat_head[itm.lh] = s.tile_mass[0];
                    last = 1;
                } else {
                    for (int rr = 0; rr < itm.nr; ++rr) {
                        stat_part[(size_t)itm.lh * T + Item::pick(itm.t, rr)] =
                            s.tile_mass[itm.nr == 2 ? rr : 0];
                        __threadfence();
                        if (atomicAdd(&tickets[itm.lh], 1u) == (unsigned)(T - 1)) last = 1;
                    }
                }
                s.head_last = last;
            }
            tc::named_bar_sync(1, NSOFT);
            if (s.head_last) {
                __threadfence();
                if (T > 1) {
                    for (int vv = sid; vv < p.N_v; vv += NSOFT) {
                        float a = 0.f;
                        for (int tt = 0; tt < T; ++tt)
                            a += __ldcg(&score_part[((size_t)itm.lh * T + tt) * p.N_v + vv]);
                        scores[(size_t)itm.lh * p.N_v + vv] = a;
                    }
                    if (sid == 0) {
                        float a = 0.f;
                        for (int tt = 0; tt < T; ++tt) a += __ldcg(&stat_part[(size_t)itm.lh * T + tt]);
                        stat_head[itm.lh] = a;
                        tickets[itm.lh] = 0u;
                    }
                }
                if (sid == 0) {
                    __threadfence();
                    if (atomicAdd(&tickets[p.L * p.H_kv + itm.l], 1u) == (unsigned)(p.H_kv - 1)) {
                        __threadfence();
                        float S = 0.f;
                        for (int gg = 0; gg < p.H_kv; ++gg)
                            S += __ldcg(&stat_head[(size_t)itm.l * p.H_kv + gg]);
                        tvb_stat[itm.l] = S;
                        tickets[p.L * p.H_kv + itm.l] = 0u;
                    }
                }
            }
            const bool stop = s.stop;
            if (stop) break;
        }
        if (!ok) raise_status(status, TGVKV_STATUS_TIMEOUT);
    }

    // ------------------------------------------------------------ teardown
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, TMEM_COLS);
    }
}

// ---- host: tensor maps ------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

// [rows][d] bf16, boxes of 64 x box_rows, 128-byte swizzle
bool make_map(CUtensorMap* map, const void* base, uint64_t rows, int d, uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
    const cuuint32_t box[2] = {64, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
    static int counts[64] = {};
    static std::mutex mu;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!counts[dev]) cudaDeviceGetAttribute(&counts[dev], cudaDevAttrMultiProcessorCount, dev);
    return counts[dev];
}

template <int D>
cudaError_t launch_tc(const Problem& p, const uint16_t* q, const uint16_t* k,
                      const uint8_t* modality, const int32_t* text_pos, const float* w,
                      float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                      cudaStream_t stream) {
    alignas(64) CUtensorMap mq, mk;
    if (!make_map(&mq, q, (uint64_t)p.L * p.H_q * p.n_win, D, 32) ||
        !make_map(&mk, k, (uint64_t)p.L * p.H_kv * p.N, D, BN))
        return cudaErrorInvalidValue;
    static_assert(sizeof(PSmem<D>) + 1024 <= 227 * 1024, "shared memory of one CTA");
    const size_t smem = sizeof(PSmem<D>) + 1024;
    cudaError_t e = cudaFuncSetAttribute(score_tc_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(score_tc_kernel<D>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    const int npair = p.T >= 2 ? (p.T + 1) / 2 : 1;
    const int n_items = p.L * p.H_kv * npair;
    const int sms = sm_count();
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int grid = n_items < sms ? n_items : sms;
    score_tc_kernel<D><<<grid, NTHREADS, smem, stream>>>(
        mq, mk, p, modality, text_pos, w, scores, tvb_stat,
        reinterpret_cast<float*>(ws + lay.score_part), reinterpret_cast<float*>(ws + lay.stat_part),
        reinterpret_cast<float*>(ws + lay.stat_head), reinterpret_cast<uint32_t*>(ws + lay.tickets),
        reinterpret_cast<uint32_t*>(ws + lay.status));
    return cudaGetLastError();
}

}  // namespace

int score_launches(const Problem& p) { return p.R == 0 ? 0 : 1; }

cudaError_t launch_score(const Problem& p, const uint16_t* q, const uint16_t* k,
                         const uint8_t* modality, const int32_t* text_pos, const float* w,
                         float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                         cudaStream_t stream) {
    if (p.R == 0) {  // no query rows: no attention mass anywhere
        cudaError_t e = cudaSuccess;
        if (p.N_v > 0)
            e = cudaMemsetAsync(scores, 0, sizeof(float) * (size_t)p.L * p.H_kv * p.N_v, stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(tvb_stat, 0, sizeof(float) * (size_t)p.L, stream);
        return e;
    }
    if (p.d == 64)
        return launch_tc<64>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
    return launch_tc<128>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
}

}  // namespace tgvkv
