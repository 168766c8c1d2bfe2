// TWR scores and TVB statistic on the 5th-generation tensor cores (tcgen05):
// a persistent, warp-specialised kernel with one CTA per SM.
//
// The query rows of one (layer, KV head) -- the G query heads of the group
// stacked over the n_win text-query rows -- form 128-row tiles.  Every row
// streams the head's keys twice, the two passes of Eq. 2 / Eq. 8:
//
//   pass A  S = Q K^T  (TMEM lane = query row): per row an online maximum m_i,
//           normaliser Z_i and vision mass V_i over every visible key (causal:
//           key j <= position of row i).
//   pass B  S^T = K Q^T  (TMEM lane = key) over the key tiles that hold vision
//           keys: per key j the sum over rows of c_i 2^(x_ij - m_i),
//           c_i = w_i / (G Z_i) -- the text-weighted column sum of Eq. 8 with
//           the GQA mean folded in.  c_i goes into the exponent,
//           2^(x_ij - m'_i) with m'_i = m_i - log2 c_i, so a term is one
//           FFMA, one EX2 and one FADD, and no cross-lane reduction is needed.
//
// The pipeline moves in steps; a step fills one of two 256-column fp32 TMEM
// accumulators, and all 16 softmax warps consume every step.  What a step
// holds depends on the shape of the work item:
//
//   pair    (a head with 2+ row tiles; an item is two row tiles of one head)
//           one K tile x both row tiles.  Pass A: columns [128r, 128r+128) =
//           Q_r K^T.  Pass B: one N = 256 product K [Q_0; Q_1]^T.  Each K tile
//           is read once for 256 query rows.
//   single  (one row tile of more than 64 rows) two K tiles x the row tile.
//   packed  (one row tile of at most 64 rows) TWO heads share the 128 lanes:
//           head h's rows live in lane quarters 2h and 2h+1, and a step holds
//           one K tile of each head; columns [128h, 128h+128) are
//           [Q_0; Q_1] K_h^T, of which only head h's lanes are read (pass A),
//           and K_h [Q_0; Q_1]^T, of which only head h's columns are read
//           (pass B).  Every lane and every softmax thread does useful work.
//           Two-head items fill whole rounds of the grid; the remaining heads
//           are one-head items, so the last round spreads over more CTAs.
//
// Roles: warp 0 fetches items from a global counter (longest first) and issues
// TMA loads -- an item's Q rows, then every K tile of both passes through a
// 4-stage ring; warps 1 and 18 issue the MMAs of alternate steps (a thread
// that waits on an mbarrier lets its own MMA queue drain, so two issuers keep
// the tensor pipe busy; step k always uses accumulator k & 1, so each issuer
// owns one accumulator); warp 1 also owns the 512 TMEM columns; warps 2-17 run
// the softmax, four per TMEM lane quarter.  Every wait is bounded (about 1 s
// of SM cycles); a timeout sets TGVKV_STATUS_TIMEOUT and the CTA unwinds.
//
// With Problem::keys_text set, pass B runs over the text keys with unit row
// weights (c_i = 1 / (G Z_i)): the text scores of Eq. 9.  The launcher then
// passes N_t as the key-set size in N_v.
//
// Results do not depend on the schedule: every key's pass-B sum is two
// partial sums added onto zero (the same in either order); the row tiles of a
// head write partial score rows that the last pair to finish adds in tile
// order; and the last CTA to finish adds the per-head TV masses of each layer
// in head order.
#include <cudaTypedefs.h>
#include <limits.h>
#include <math.h>

#include <mutex>

#include "budget.cuh"
#include "common.cuh"
#include "launch.h"
#include "rowstat.cuh"
#include "tc05.cuh"

namespace tgvkv {
namespace {

constexpr int BM = 128;           // query rows per row tile = TMEM lanes
constexpr int BN = 128;           // keys per K tile
constexpr int STAGES = 4;         // K tiles in flight
constexpr int NIQ = 2;            // items fetched ahead
constexpr int NSW = 16;           // softmax warps (4 per TMEM lane quarter)
constexpr int NSOFT = NSW * 32;
constexpr int MMA2_WARP = 2 + NSW;
constexpr int NTHREADS = (NSW + 3) * 32;
constexpr int SCOLS = 256;        // accumulator columns per step
constexpr int TMEM_COLS = 2 * SCOLS;
constexpr int MAXT = kMaxN / BN;  // key tiles per head
constexpr int MAX_RT = 256;       // row tiles per KV head (G * n_win <= 32768)
constexpr uint32_t IDESC128 = tc::idesc_bf16(128, 128);
constexpr uint32_t IDESC256 = tc::idesc_bf16(128, 256);
constexpr uint32_t IDESC64 = tc::idesc_bf16(128, 64);

enum { MODE_PAIR = 0, MODE_SINGLE = 1, MODE_PACKED = 2 };

template <int D>
struct PSmem {
    uint16_t q[D / 64][2][BM * 64];          // two Q slots; per 64 dims, 128-byte-swizzled rows
    // K ring, stage-major within each 64 dims, so that the rows of stages 2j and
    // 2j+1 are adjacent: single and packed steps multiply both in one N = 256 MMA
    uint16_t k[D / 64][STAGES][BN * 64];
    uint64_t full[STAGES], empty[STAGES];
    uint64_t s_full[2], s_empty[2];
    uint64_t q_full[2], q_empty[2], mma_done;
    uint64_t it_full[NIQ], it_empty[NIQ];
    uint32_t vmask[MAXT][4];                 // vision bit of each key of each tile
    int vis_before[MAXT + 1];                // vision keys before each tile
    int vq[MAXT][4];                         // vision keys before each 32-key word
    int rt_max[MAX_RT], rt_min[MAX_RT];      // per row tile: max / min query position
    alignas(16) int row_pos[2][BM];          // per row slot and TMEM lane: position, -1 = none
    int row_q[2][BM];                        // ... its global Q row, -1 = none
    alignas(16) float row_nmp[2][BM];        // -(m_i - log2 c_i); -inf = no row
    float row_w[2][BM], row_mass[2][BM];
    float part_m[4][BM], part_z[4][BM], part_v[4][BM], part_u[4][BM];
    int item_q[NIQ];
    uint32_t tmem_base;
    int abort_flag, never, stop, head_last, cur_item, cta_last;
    float tile_mass[2];
};

// One work item.  "part" 0/1 is a row tile (pair) or a head (packed); a single
// item has part 0 only.
struct Item {
    int lh[2], l[2];          // (layer, KV head) of each part; lh[1] < 0: absent
    int qy[2];                // first global Q row of each part's rows
    int rows[2], rpg[2];      // rows of each part, and rows per 32-lane group
    int nt[2], minp[2];       // pass-A key tiles and least query position of each part
    int ntmax, nparts, pidx;  // pidx: which pair of the head (pair items)
    __device__ __forceinline__ static int pick(const int (&a)[2], int r) { return r ? a[1] : a[0]; }
};

__device__ __forceinline__ int next_vis_tile(const int* vis_before, int kt, int n_tiles) {
    while (kt < n_tiles && vis_before[kt + 1] == vis_before[kt]) ++kt;
    return kt;
}

// First global Q row of the 32-row box that lands in TMEM lanes 32g..32g+31
// of Q slot r: pair / single -> part r's rows g*rpg..; packed -> head g/2's
// rows (g%2)*rpg.. (an absent second head repeats the first's).
__device__ __forceinline__ int q_box_row(const Item& it, int mode, int r, int g) {
    if (mode == MODE_PACKED) {
        const int h = (g >> 1) < it.nparts ? (g >> 1) : 0;
        return Item::pick(it.qy, h) + (g & 1) * it.rpg[0];
    }
    return Item::pick(it.qy, r) + g * Item::pick(it.rpg, r);
}

// n_two: packed launches only -- items below n_two hold two heads, the rest
// one head each (the last round of a launch, so that it spreads over more CTAs).
template <int D>
__device__ __forceinline__ Item item_info(const Problem& p, const PSmem<D>& s, int mode, int id,
                                          int n_two) {
    Item it;
    const int LH = p.L * p.H_kv;
    it.pidx = 0;
    if (mode == MODE_PAIR) {
        const int npair = score_pairs(p);
        const int lh = id / npair;
        const int tp = npair - 1 - id % npair;   // later row tiles (longer causal range) first
        it.pidx = tp;
        const int t0 = 2 * tp, t1 = 2 * tp + 1 < p.T ? 2 * tp + 1 : -1;
        it.nparts = t1 >= 0 ? 2 : 1;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int t = r == 0 ? t0 : (t1 >= 0 ? t1 : t0);
            it.lh[r] = (r == 0 || t1 >= 0) ? lh : -1;
            it.l[r] = lh / p.H_kv;
            it.qy[r] = (it.l[r] * p.H_q + (lh % p.H_kv) * p.G) * p.n_win + t * BM;
            it.rows[r] = min(BM, p.R - t * BM);
            it.rpg[r] = (it.rows[r] + 3) >> 2;
            it.nt[r] = (s.rt_max[t] + BN) / BN;
            it.minp[r] = s.rt_min[t];
        }
    } else {
        const bool packed = mode == MODE_PACKED;
        const bool two = packed && id < n_two;
        const int first = !packed ? id : (two ? 2 * id : n_two + id);
        it.nparts = 1;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int lh = first + r;
            it.lh[r] = (r == 0 || (two && lh < LH)) ? lh : -1;
            if (it.lh[r] >= 0 && r == 1) it.nparts = 2;
            const int lhv = it.lh[r] >= 0 ? lh : first;
            it.l[r] = lhv / p.H_kv;
            it.qy[r] = (it.l[r] * p.H_q + (lhv % p.H_kv) * p.G) * p.n_win;
            it.rows[r] = p.R;
            it.rpg[r] = packed ? (p.R + 1) >> 1 : (p.R + 3) >> 2;
            it.nt[r] = (s.rt_max[0] + BN) / BN;
            it.minp[r] = s.rt_min[0];
        }
    }
    it.ntmax = it.nparts == 2 ? max(it.nt[0], it.nt[1]) : it.nt[0];
    return it;
}

// Key tiles of the next step of a pass (0 = A, 1 = B); false at the end.
// kt[1] is the second tile of a single step or the second head's tile of a
// packed step (-1: none); pair steps use kt[0] for both row tiles.
__device__ __forceinline__ bool next_step(const Item& it, int mode, int pass, int& cur,
                                          const int* vis_before, int (&kt)[2], bool stats_given) {
    if (pass == 0 && stats_given) return false;   // the row statistics come from the workspace
    int c = pass == 0 ? cur : next_vis_tile(vis_before, cur, it.ntmax);
    if (c >= it.ntmax) return false;
    kt[0] = c;
    cur = c + 1;
    kt[1] = -1;
    if (mode == MODE_SINGLE) {
        const int c2 = pass == 0 ? cur : next_vis_tile(vis_before, cur, it.ntmax);
        if (c2 < it.ntmax) {
            kt[1] = c2;
            cur = c2 + 1;
        }
    } else if (mode == MODE_PACKED && it.lh[1] >= 0) {
        kt[1] = c;
    }
    return true;
}

// Sum over the valid rows of one 32-row group of 2^(y_i sl2 + nmp_i), with the
// causal mask j <= pos_i.  FULL: all 32 rows exist; ALL_VIS: every row sees
// key j (no mask; a template argument, so that the unrolled loop has no
// branch on it).
template <bool FULL, bool ALL_VIS>
__device__ __forceinline__ float colsum_group(const float (&y)[32], const float* nmp,
                                              const int* pos, float sl2, int rpg, int j) {
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
            if (!ALL_VIS) {
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

// A bounded wait whose outcome is the same for every lane of the warp (the
// tensor-memory loads that follow are warp-collective).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, abort);
    return __all_sync(~0u, got);
}

// D/16 MMAs of one 128-row x N-column product, K = D in steps of 16.  a / b
// are the descriptors of the operands' first 64-dim half; a 64-dim half of an
// operand lies a_half / b_half 16-byte units further (the 32-byte K step
// inside a 128-byte swizzle atom is 2 units).
template <int D>
__device__ __forceinline__ void mma_block(uint32_t d_tmem, uint64_t a, uint32_t a_half, uint64_t b,
                                          uint32_t b_half, uint32_t idesc) {
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t ka = a + (uint64_t)((kk >> 2) * a_half + (kk & 3) * 2);
        const uint64_t kb = b + (uint64_t)((kk >> 2) * b_half + (kk & 3) * 2);
        if (kk == 0)
            tc::mma_bf16_c<0>(d_tmem, ka, kb, idesc);
        else
            tc::mma_bf16_c<1>(d_tmem, ka, kb, idesc);
    }
}

// Release this warp's claim on a step accumulator (after its tensor-memory
// loads have completed).
__device__ __forceinline__ void release_acc(uint64_t* bar, int lane) {
    tc::fence_before_sync();
    __syncwarp();
    if (lane == 0) tc::mbar_arrive(bar);
}

template <int D, int MODE>
__global__ void __launch_bounds__(NTHREADS, 1)
score_tc_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                Problem p, int n_items, int n_two, const uint8_t* __restrict__ modality,
                const int32_t* __restrict__ text_pos, const float* __restrict__ w,
                float* __restrict__ scores, float* __restrict__ tvb_stat,
                float* __restrict__ score_part, float* __restrict__ stat_part,
                float* __restrict__ stat_head, uint32_t* __restrict__ tickets,
                uint32_t* __restrict__ status, long long budget_total, int32_t* __restrict__ budgets) {
    float* row_stats = p.row_stats;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    PSmem<D>& s = *reinterpret_cast<PSmem<D>*>(smem_raw + (((raw + 1023u) & ~1023u) - raw));
    constexpr uint32_t KTILE_BYTES = (D / 64) * BN * 128;
    constexpr uint32_t QBOX_BYTES = 32 * 128;            // 32 rows x 64 dims
    constexpr uint32_t K_HALF = STAGES * BN * 64 * 2 / 16;   // 64-dim half of the K ring, 16-byte units
    constexpr uint32_t Q_HALF = 2 * BM * 64 * 2 / 16;    // 64-dim half of the Q slots
    constexpr uint32_t Q_SLOT = BM * 64 * 2 / 16;

    constexpr int mode = MODE;   // the item shape, fixed per launch
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const float sl2 = p.scale_log2;
    const int LH = p.L * p.H_kv;
    uint32_t* work_counter = tickets + LH;
    uint32_t* done_counter = work_counter + 1;
    uint32_t* exit_counter = work_counter + 2;

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
        for (int i = 0; i < STAGES; ++i) {
            tc::mbar_init(&s.full[i], 1);
            tc::mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&s.s_full[i], 1);
            tc::mbar_init(&s.s_empty[i], NSW);   // one arrival per softmax warp
            tc::mbar_init(&s.q_full[i], 1);
            tc::mbar_init(&s.q_empty[i], 2);     // both MMA issuers
        }
        for (int i = 0; i < NIQ; ++i) {
            tc::mbar_init(&s.it_full[i], 1);
            tc::mbar_init(&s.it_empty[i], 3);    // the two MMA issuers and the softmax role
        }
        tc::mbar_init(&s.mma_done, 2);
        tc::fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&s.tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    const int n_tiles_all = (p.N + BN - 1) / BN;
    // the first row positions are loaded now, so that their latency overlaps
    // the modality loads below
    const int pos0 = tid < p.R ? text_pos[tid % p.n_win] : -1;
    for (int kt = warp; kt < n_tiles_all; kt += NTHREADS / 32) {
        int cnt = 0;
#pragma unroll
        for (int wd = 0; wd < 4; ++wd) {
            const int j = kt * BN + wd * 32 + lane;
            // the key set of pass B: vision keys, or text keys (Eq. 9)
            const unsigned m = __ballot_sync(~0u, j < p.N && (modality[j] != 0) != (p.keys_text != 0));
            if (lane == 0) {
                s.vmask[kt][wd] = m;
                s.vq[kt][wd] = cnt;              // within the tile, for now
            }
            cnt += __popc(m);
        }
        if (lane == 0) s.vis_before[kt] = cnt;
    }
    for (int t = tid; t < p.T; t += NTHREADS) {
        s.rt_max[t] = -1;
        s.rt_min[t] = INT_MAX;
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    for (int r = tid; r < p.R; r += NTHREADS) {
        const int pos = r == tid ? pos0 : text_pos[r % p.n_win];
        if (pos >= 0 && pos < p.N) {
            atomicMax(&s.rt_max[r / BM], pos);
            atomicMin(&s.rt_min[r / BM], pos);
        }
    }
    if (warp == 0) {
        // exclusive scan of the per-tile vision counts
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
    for (int kt = tid; kt < n_tiles_all; kt += NTHREADS)
#pragma unroll
        for (int wd = 0; wd < 4; ++wd) s.vq[kt][wd] += s.vis_before[kt];
    __syncthreads();
    const uint32_t tmem = s.tmem_base;
    volatile int* abort_flag = &s.abort_flag;

    // ------------------------------------------------------------ producer
    // Items are claimed from a counter in order, longest first (pair items
    // differ in length); CTA c starts with item c without a claim.
    if (warp == 0 && lane == 0) {
        tc::tma_prefetch_desc(&tmap_q);
        tc::tma_prefetch_desc(&tmap_k);
        int it = 0;
        int qn0 = 0, qn1 = 0;     // uses of each Q slot
        bool ok = true;
        for (int n = 0; ok; ++n) {
            // fetch the next item (or the end mark) for every role of this CTA
            const int slot = n % NIQ;
            if (!tc::mbar_wait(&s.it_empty[slot], ((n / NIQ) & 1) ^ 1, abort_flag)) {
                ok = false;
                break;
            }
            // the first item of CTA c is item c (grid <= items); later ones are claimed
            const int id = n == 0 ? (int)blockIdx.x : (int)gridDim.x + (int)atomicAdd(work_counter, 1u);
            s.item_q[slot] = id < n_items ? id : -1;
            tc::mbar_arrive(&s.it_full[slot]);
            if (id >= n_items) {
                // the last CTA to run out of work re-arms the counter for the next launch
                if (atomicAdd(done_counter, 1u) == gridDim.x - 1) {
                    *work_counter = 0u;
                    *done_counter = 0u;
                }
                break;
            }
            const Item itm = item_info(p, s, mode, id, n_two);
            // Q rows: pair items fill both slots (row tile r -> slot r); single
            // and packed items alternate slots.  Four boxes of 32 rows per slot,
            // box g landing in TMEM lanes 32g..32g+31.
            const int nslot = mode == MODE_PAIR ? itm.nparts : 1;
            for (int r = 0; r < nslot; ++r) {
                const int qs = mode == MODE_PAIR ? r : (n & 1);
                const int use = qs ? qn1++ : qn0++;
                if (!tc::mbar_wait(&s.q_empty[qs], (use & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::mbar_arrive_expect_tx(&s.q_full[qs], 4 * (D / 64) * QBOX_BYTES);
#pragma unroll
                for (int qg = 0; qg < 4; ++qg) {
                    const int y = q_box_row(itm, mode, r, qg);
#pragma unroll
                    for (int h = 0; h < D / 64; ++h)
                        tc::tma_load_2d(&s.q[h][qs][qg * 32 * 64], &tmap_q, h * 64, y, &s.q_full[qs]);
                }
            }
            auto load = [&](int lh, int kt) {
                const int stage = it % STAGES;
                if (!tc::mbar_wait(&s.empty[stage], ((it / STAGES) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    return;
                }
                tc::mbar_arrive_expect_tx(&s.full[stage], KTILE_BYTES);
#pragma unroll
                for (int h = 0; h < D / 64; ++h)
                    tc::tma_load_2d(&s.k[h][stage][0], &tmap_k, h * 64, lh * p.N + kt * BN,
                                    &s.full[stage]);
                ++it;
            };
            // a stage a step does not use (single / packed steps always take two)
            auto skip = [&]() {
                const int stage = it % STAGES;
                if (!tc::mbar_wait(&s.empty[stage], ((it / STAGES) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    return;
                }
                tc::mbar_arrive(&s.full[stage]);
                ++it;
            };
            for (int pass = 0; ok && pass < 2; ++pass) {
                int cur = 0, kt[2];
                while (ok && next_step(itm, mode, pass, cur, s.vis_before, kt, p.stats_given)) {
                    load(itm.lh[0], kt[0]);
                    if (ok && kt[1] >= 0)
                        load(mode == MODE_PACKED ? itm.lh[1] : itm.lh[0], kt[1]);
                    else if (ok && mode != MODE_PAIR)
                        skip();
                }
            }
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every copy this CTA issued has landed before it may exit
        if (qn0 > 0) tc::mbar_wait(&s.q_full[0], (qn0 - 1) & 1, &s.never);
        if (qn1 > 0) tc::mbar_wait(&s.q_full[1], (qn1 - 1) & 1, &s.never);
        for (int i = max(0, it - STAGES); i < it; ++i)
            tc::mbar_wait(&s.full[i % STAGES], (i / STAGES) & 1, &s.never);
    }

    // ------------------------------------------------------------ MMA issuers
    // Step k goes to issuer k & 1 and accumulator k & 1.
    if ((warp == 1 || warp == MMA2_WARP) && lane == 0) {
        const int me = warp == 1 ? 0 : 1;
        // shared-memory descriptors, computed once: the start-address field
        // (16-byte units, < 2^14 inside 256 KB) takes plain additions
        const uint64_t kdesc0 = tc::sdesc_k_sw128(smem_u32(&s.k[0][0][0]));
        const uint64_t qdesc0 = tc::sdesc_k_sw128(smem_u32(&s.q[0][0][0]));
        constexpr uint32_t KSTAGE_DESC = BN * 64 * 2 / 16;   // one stage within a 64-dim half
        int it = 0, step = 0;
        int qn0 = 0, qn1 = 0;     // uses of each Q slot
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
            const Item itm = item_info(p, s, mode, id, n_two);
            const int nslot = mode == MODE_PAIR ? itm.nparts : 1;
            const int qs0 = mode == MODE_PAIR ? 0 : (n & 1);
            for (int r = 0; r < nslot; ++r) {
                const int qs = mode == MODE_PAIR ? r : qs0;
                const int use = qs ? qn1++ : qn0++;
                if (!tc::mbar_wait(&s.q_full[qs], use & 1, abort_flag)) {
                    ok = false;
                    break;
                }
            }
            if (!ok) break;
            const uint64_t qd = qdesc0 + (uint64_t)(qs0 * Q_SLOT);
            for (int pass = 0; ok && pass < 2; ++pass) {
                int cur = 0, kt[2];
                while (ok && next_step(itm, mode, pass, cur, s.vis_before, kt, p.stats_given)) {
                    // pair steps take one stage; single and packed steps two (an even
                    // pair of adjacent stages), the second possibly unused
                    const int nst = mode == MODE_PAIR ? 1 : 2;
                    const bool has2 = kt[1] >= 0;
                    if ((step & 1) == me) {
                        const int b = step & 1;
                        bool got = tc::mbar_wait(&s.full[it % STAGES], (it / STAGES) & 1, abort_flag);
                        if (got && nst == 2)
                            got = tc::mbar_wait(&s.full[(it + 1) % STAGES], ((it + 1) / STAGES) & 1,
                                                abort_flag);
                        if (got) got = tc::mbar_wait(&s.s_empty[b], ((step >> 1) & 1) ^ 1, abort_flag);
                        if (!got) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        const uint32_t d = tmem + (uint32_t)(b * SCOLS);
                        const uint64_t k0 = kdesc0 + (uint64_t)((it % STAGES) * KSTAGE_DESC);
                        const uint64_t k1 = kdesc0 + (uint64_t)(((it + 1) % STAGES) * KSTAGE_DESC);
                        if (mode == MODE_PAIR) {
                            if (pass == 0) {
                                if (kt[0] < itm.nt[0])
                                    mma_block<D>(d, qd, Q_HALF, k0, K_HALF, IDESC128);
                                if (itm.nparts == 2 && kt[0] < itm.nt[1])
                                    mma_block<D>(d + BN, qd + Q_SLOT, Q_HALF, k0, K_HALF, IDESC128);
                            } else if (itm.nparts == 2) {
                                mma_block<D>(d, k0, K_HALF, qd, Q_HALF, IDESC256);
                            } else {
                                mma_block<D>(d, k0, K_HALF, qd, Q_HALF, IDESC128);
                            }
                        } else if (pass == 0) {
                            // Q against both adjacent K stages in one N = 256 product
                            mma_block<D>(d, qd, Q_HALF, k0, K_HALF, has2 ? IDESC256 : IDESC128);
                        } else if (mode == MODE_PACKED) {
                            // head h's rows are Q rows 64h..64h+63 (64 rows = 8 KB = 512 units on)
                            mma_block<D>(d, k0, K_HALF, qd, Q_HALF, IDESC64);
                            if (has2) mma_block<D>(d + BN + 64, k1, K_HALF, qd + 512, Q_HALF, IDESC64);
                        } else {
                            mma_block<D>(d, k0, K_HALF, qd, Q_HALF, IDESC128);
                            if (has2) mma_block<D>(d + BN, k1, K_HALF, qd, Q_HALF, IDESC128);
                        }
                        tc::mma_commit(&s.s_full[b]);
                        tc::mma_commit(&s.empty[it % STAGES]);
                        if (nst == 2) tc::mma_commit(&s.empty[(it + 1) % STAGES]);
                    }
                    it += nst;
                    ++step;
                }
            }
            // the item's Q slots are free once both issuers' MMAs have finished
            for (int r = 0; r < nslot; ++r) tc::mma_commit(&s.q_empty[mode == MODE_PAIR ? r : qs0]);
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
    if (warp >= 2 && warp < MMA2_WARP) {
        // The kernel before (the select + gather of the previous eviction, when it
        // is one) may still read the scores and budgets this kernel overwrites: the
        // softmax role, the only one writing global memory before the end, waits
        // for it.  The loads and MMAs of the first items overlap its end.
        griddep_wait();
        const int sid = tid - 64;
        const int quarter = warp & 3;
        const int wi = (warp - 2) >> 2;                     // 0..3 within the lane quarter
        const int ln = quarter * 32 + lane;                 // this thread's TMEM lane
        const uint32_t tq = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t lt_mask = (1u << lane) - 1u;
        int step = 0;
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
            const Item itm = item_info(p, s, mode, id, n_two);

            // ---- rows: lane 32q + i of row slot rs holds the part's row q*rpg + i
            // (packed: lanes 64h + 32q' + i hold head h's row q'*rpg + i)
            if (wi < (mode == MODE_PAIR ? itm.nparts : 1)) {
                const int rs = wi;
                int part, row;
                if (mode == MODE_PACKED) {
                    part = quarter >> 1;
                    row = (quarter & 1) * itm.rpg[0] + lane;
                } else {
                    part = rs;
                    row = quarter * Item::pick(itm.rpg, rs) + lane;
                }
                int pos = -1;
                float wr = 0.f;
                const bool has = lane < Item::pick(itm.rpg, part) && row < Item::pick(itm.rows, part) &&
                                 Item::pick(itm.lh, part) >= 0;
                if (has) {
                    const int t_row = mode == MODE_PAIR ? (2 * itm.pidx + rs) * BM : 0;
                    const int wi_row = (t_row + row) % p.n_win;
                    pos = text_pos[wi_row];
                    if (pos < 0 || pos >= p.N) pos = -1;
                    if (p.keys_text) {
                        wr = 1.f;   // Eq. 9: unweighted column sums
                    } else {
                        wr = w[(long long)Item::pick(itm.l, part) * p.w_stride + wi_row];
                        if (!(wr >= 0.f) || isinf(wr)) {
                            raise_status(status, TGVKV_STATUS_WEIGHT);
                            wr = 0.f;
                        }
                    }
                }
                s.row_pos[rs][ln] = pos;
                s.row_w[rs][ln] = wr;
                s.row_q[rs][ln] = has ? Item::pick(itm.qy, part) + row : -1;
            }
            // the item's output rows start at zero: pass B adds two partial sums per key
            for (int r = 0; r < itm.nparts; ++r) {
                float* out = mode == MODE_PAIR
                                 ? score_part + ((size_t)itm.lh[0] * p.T + 2 * itm.pidx + r) * p.N_v
                                 : scores + (size_t)Item::pick(itm.lh, r) * p.N_v;
                for (int vv = sid; vv < p.N_v; vv += NSOFT) out[vv] = 0.f;
            }
            tc::named_bar_sync(1, NSOFT);

            // ---- pass A: this warp's share of each step
            // pair: row tile r = wi >> 1, columns 128r + 64(wi & 1) + [0, 64)
            // single: K tile b = wi >> 1, columns 128b + 64(wi & 1) + [0, 64)
            // packed: head b = quarter >> 1, columns 128b + 32 wi + [0, 32)
            const int rsA = mode == MODE_PAIR ? (wi >> 1) : 0;
            const int my_pos = s.row_pos[rsA][ln];
            float m = -INFINITY, z = 0.f, v = 0.f, u = 0.f;
            {
                // Every warp runs every step of the item, also after a failed wait
                // (then doing nothing), so that the warps of a quarter always meet
                // at the same named barriers.
                int cur = 0, kt[2];
                while (next_step(itm, mode, 0, cur, s.vis_before, kt, p.stats_given)) {
                    const int b = step & 1;
                    ++step;
                    if (ok && !warp_wait(&s.s_full[b], ((step - 1) >> 1) & 1, abort_flag)) {
                        ok = false;
                        s.abort_flag = 1;
                    }
                    if (!ok) continue;
                    tc::fence_after_sync();
                    int blk, ktile, cbase, nch;
                    bool act;
                    if (mode == MODE_PAIR) {
                        blk = wi >> 1;
                        ktile = kt[0];
                        act = blk < itm.nparts && ktile < Item::pick(itm.nt, blk);
                        cbase = 64 * (wi & 1);
                        nch = 2;
                    } else if (mode == MODE_SINGLE) {
                        blk = wi >> 1;
                        ktile = Item::pick(kt, blk);
                        act = ktile >= 0;
                        cbase = 64 * (wi & 1);
                        nch = 2;
                    } else {
                        blk = quarter >> 1;
                        ktile = Item::pick(kt, blk);
                        act = ktile >= 0;
                        cbase = 32 * wi;
                        nch = 1;
                    }
                    if (!act) {
                        release_acc(&s.s_empty[b], lane);
                    } else {
                        const uint32_t ta = tq + (uint32_t)(b * SCOLS + blk * BN + cbase);
                        for (int ch = 0; ch < nch; ++ch) {
                            float x[32];
                            tc::tmem_ld32(ta + (uint32_t)(ch * 32), x);
                            tc::tmem_wait_ld();
                            if (ch == nch - 1) release_acc(&s.s_empty[b], lane);
                            const int lim = my_pos - (ktile * BN + cbase + ch * 32);
                            const uint32_t vm = s.vmask[ktile][(cbase >> 5) + ch];
                            if (p.keys_text)   // also the vision mass, for the vision pass
                                row_word_both(x, sl2, lim, vm, m, z, v, u);
                            else
                                row_word(x, sl2, lim, vm, m, z, v);
                        }
                    }
                }
            }

            // ---- combine the partial statistics of each row
            s.part_m[wi][ln] = m;
            s.part_z[wi][ln] = z;
            s.part_v[wi][ln] = v;
            s.part_u[wi][ln] = u;
            tc::named_bar_sync(2 + quarter, 128);
            // pair: warps 0 and 2 combine parts {0,1} / {2,3} of row slot 0 / 1;
            // single and packed: warp 0 combines all four
            if (mode == MODE_PAIR ? ((wi & 1) == 0 && (wi >> 1) < itm.nparts) : wi == 0) {
                const int rs = mode == MODE_PAIR ? (wi >> 1) : 0;
                const int c0 = mode == MODE_PAIR ? wi : 0, c1 = mode == MODE_PAIR ? wi + 2 : 4;
                const int qr = s.row_q[rs][ln];
                float mt = -INFINITY;
                float zt = 0.f, vt = 0.f;
                if (p.stats_given) {
                    // (m, Z, vision mass) of the row, from the text-key pass
                    if (qr >= 0) {
                        mt = __ldcg(row_stats + 3 * (size_t)qr);
                        zt = __ldcg(row_stats + 3 * (size_t)qr + 1);
                        vt = __ldcg(row_stats + 3 * (size_t)qr + 2);
                    }
                } else {
                    for (int c = c0; c < c1; ++c) mt = fmaxf(mt, s.part_m[c][ln]);
                    float ut = 0.f;
                    if (mt != -INFINITY) {
                        for (int c = c0; c < c1; ++c) {
                            const float a = fast_exp2(s.part_m[c][ln] - mt);
                            zt += s.part_z[c][ln] * a;
                            vt += s.part_v[c][ln] * a;
                            ut += s.part_u[c][ln] * a;
                        }
                    }
                    if (p.keys_text && row_stats && qr >= 0) {
                        row_stats[3 * (size_t)qr] = mt;
                        row_stats[3 * (size_t)qr + 1] = zt;
                        row_stats[3 * (size_t)qr + 2] = ut;
                    }
                }
                const bool valid = s.row_pos[rs][ln] >= 0 && zt > 0.f;
                // rows without attention get -m' = -inf: every term 2^-inf = 0
                s.row_nmp[rs][ln] =
                    valid ? fast_log2(s.row_w[rs][ln] / ((float)p.G * zt)) - mt : -INFINITY;
                s.row_mass[rs][ln] = valid ? vt / zt : 0.f;
            }
            tc::named_bar_sync(1, NSOFT);
            if (sid < 64) {
                // TV mass of each part, in lane order: pair -> row slot r over all
                // lanes; packed -> head h over lanes 64h..64h+63; single -> all lanes
                const int r = sid >> 5;
                float a = 0.f;
                if (mode == MODE_PAIR) {
                    if (r < itm.nparts)
                        a = (s.row_mass[r][lane] + s.row_mass[r][lane + 32]) +
                            (s.row_mass[r][lane + 64] + s.row_mass[r][lane + 96]);
                } else if (mode == MODE_PACKED) {
                    a = s.row_mass[0][64 * r + lane] + s.row_mass[0][64 * r + 32 + lane];
                } else if (r == 0) {
                    a = (s.row_mass[0][lane] + s.row_mass[0][lane + 32]) +
                        (s.row_mass[0][lane + 64] + s.row_mass[0][lane + 96]);
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(~0u, a, o);
                if (lane == 0) s.tile_mass[r] = a;
            }

            // ---- pass B: text-weighted column sums, one key per lane
            // pair: columns 64 wi + [0, 64) of the N = 256 product (row slot wi >> 1);
            // single: K tile b = wi >> 1, columns 128b + 64(wi & 1) + [0, 64);
            // packed: head b = wi >> 1, its rows' columns 128b + 64b + 32(wi & 1) + [0, 32).
            // Each key gets exactly two partial sums (warps 2c and 2c+1), added
            // atomically into an output row that starts at zero: 0 + a + b is the
            // same in either order, so the result does not depend on timing.
            // Pair items write one partial row per row tile.
            {
                int cur = 0, kt[2];
                while (next_step(itm, mode, 1, cur, s.vis_before, kt, p.stats_given)) {
                    const int b = step & 1;
                    if (ok && !warp_wait(&s.s_full[b], (step >> 1) & 1, abort_flag)) {
                        ok = false;
                        s.abort_flag = 1;
                    }
                    if (ok) tc::fence_after_sync();
                    int blk, ktile, ccol, rcol, rs, nch, rpg, minp;
                    bool act;
                    if (mode == MODE_PAIR) {
                        blk = 0;
                        ktile = kt[0];
                        rs = wi >> 1;
                        act = rs < itm.nparts && ktile < Item::pick(itm.nt, rs);
                        ccol = 64 * wi;
                        rcol = 64 * (wi & 1);
                        nch = 2;
                        rpg = Item::pick(itm.rpg, rs);
                        minp = Item::pick(itm.minp, rs);
                    } else if (mode == MODE_SINGLE) {
                        blk = wi >> 1;
                        ktile = Item::pick(kt, blk);
                        rs = 0;
                        act = ktile >= 0;
                        ccol = 128 * blk + 64 * (wi & 1);
                        rcol = 64 * (wi & 1);
                        nch = 2;
                        rpg = itm.rpg[0];
                        minp = itm.minp[0];
                    } else {
                        blk = wi >> 1;
                        ktile = Item::pick(kt, blk);
                        rs = 0;
                        act = ktile >= 0;
                        rcol = 64 * blk + 32 * (wi & 1);
                        ccol = 128 * blk + rcol;
                        nch = 1;
                        rpg = itm.rpg[0];
                        minp = itm.minp[0];
                    }
                    float sum = 0.f;
                    if (!ok) {
                        // unwinding: no waits, no work, but the same barriers
                    } else if (!act) {
                        release_acc(&s.s_empty[b], lane);
                    } else {
                        const int j = ktile * BN + ln;               // this lane's key
                        const bool all_vis = ktile * BN + BN - 1 <= minp;
                        const uint32_t ta = tq + (uint32_t)(b * SCOLS + ccol);
                        for (int ch = 0; ch < nch; ++ch) {
                            float y[32];
                            tc::tmem_ld32(ta + (uint32_t)(ch * 32), y);
                            tc::tmem_wait_ld();
                            if (ch == nch - 1) release_acc(&s.s_empty[b], lane);
                            const float* nmp = s.row_nmp[rs] + rcol + ch * 32;
                            const int* rp = s.row_pos[rs] + rcol + ch * 32;
                            if (rpg >= 32) {
                                if (all_vis)
                                    sum += colsum_group<true, true>(y, nmp, rp, sl2, rpg, j);
                                else
                                    sum += colsum_group<true, false>(y, nmp, rp, sl2, rpg, j);
                            } else {
                                if (all_vis)
                                    sum += colsum_group<false, true>(y, nmp, rp, sl2, rpg, j);
                                else
                                    sum += colsum_group<false, false>(y, nmp, rp, sl2, rpg, j);
                            }
                        }
                    }
                    if (ok && act) {
                        const uint32_t word = s.vmask[ktile][quarter];
                        if ((word >> lane) & 1u) {
                            const int vr = s.vq[ktile][quarter] + __popc(word & lt_mask);
                            float* out = mode == MODE_PAIR
                                             ? score_part + ((size_t)itm.lh[0] * p.T + 2 * itm.pidx + rs) * p.N_v
                                             : scores + (size_t)Item::pick(itm.lh, mode == MODE_PACKED ? blk : 0) * p.N_v;
                            if (vr < p.N_v) atomicAdd(out + vr, sum);
                        }
                    }
                    ++step;
                }
            }
            // ---- per-head results; pairs of a head meet through a ticket
            if (sid == 0) s.stop = *abort_flag;
            tc::named_bar_sync(1, NSOFT);
            if (sid == 0) {
                int last = 0;
                if (mode != MODE_PAIR) {
                    for (int h = 0; h < itm.nparts; ++h)
                        stat_head[Item::pick(itm.lh, h)] = s.tile_mass[mode == MODE_PACKED ? h : 0];
                } else {
                    for (int r = 0; r < itm.nparts; ++r)
                        stat_part[(size_t)itm.lh[0] * p.T + 2 * itm.pidx + r] = s.tile_mass[r];
                    // the barrier above ordered every thread's score writes before this fence
                    __threadfence();
                    const unsigned before = atomicAdd(&tickets[itm.lh[0]], (unsigned)itm.nparts);
                    if (before + (unsigned)itm.nparts == (unsigned)p.T) last = 1;
                }
                s.head_last = last;
            }
            tc::named_bar_sync(1, NSOFT);
            if (s.head_last) {
                // the last pair of a head adds the row tiles' partial rows in tile order
                __threadfence();
                const size_t base = (size_t)itm.lh[0] * p.T;
                for (int vv = sid; vv < p.N_v; vv += NSOFT) {
                    float a = 0.f;
                    for (int t = 0; t < p.T; ++t) a += __ldcg(&score_part[(base + t) * p.N_v + vv]);
                    scores[(size_t)itm.lh[0] * p.N_v + vv] = a;
                }
                if (sid == 0) {
                    float a = 0.f;
                    for (int t = 0; t < p.T; ++t) a += __ldcg(&stat_part[base + t]);
                    stat_head[itm.lh[0]] = a;
                    tickets[itm.lh[0]] = 0u;
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
    // the last CTA to finish adds the per-head TV masses of each layer, in head order
    if (tid == 0) {
        __threadfence();
        s.cta_last = atomicAdd(exit_counter, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    // this CTA's scores and masses are written: a programmatic dependent (the
    // select + gather of tgvkv_evict) may be scheduled once every CTA is here,
    // while the last one still splits the budgets
    griddep_launch_dependents();
    if (s.cta_last) {
        __threadfence();
        // the now idle K ring as scratch: the per-head masses, then the statistic
        float* hs = reinterpret_cast<float*>(&s.k[0][0][0]);
        const int units = p.head_budgets ? LH : p.L;
        float* us = hs + LH;
        // (the masses and the statistic take the ring's first half, the block
        // split's scratch the second; larger problems read global memory)
        const bool in_smem = (size_t)(LH + units) * sizeof(float) <= sizeof(s.k) / 2;
        // every thread loads its share of the per-head masses (one round trip)
        for (int lh = tid; lh < LH; lh += NTHREADS) {
            const float a = __ldcg(&stat_head[lh]);
            if (in_smem) hs[lh] = a;
        }
        __syncthreads();
        if (p.head_budgets) {
            // head-adaptive budgets: the statistic is the TV mass of each (layer, KV head)
            for (int lh = tid; lh < LH; lh += NTHREADS) {
                const float a = in_smem ? hs[lh] : __ldcg(&stat_head[lh]);
                tvb_stat[lh] = a;
                if (in_smem) us[lh] = a;
            }
        } else {
            // each layer's masses added in head order
            for (int l = tid; l < p.L; l += NTHREADS) {
                float S = 0.f;
                for (int g = 0; g < p.H_kv; ++g)
                    S += in_smem ? hs[(size_t)l * p.H_kv + g] : __ldcg(&stat_head[(size_t)l * p.H_kv + g]);
                tvb_stat[l] = S;
                if (in_smem) us[l] = S;
            }
        }
        __syncthreads();
        if (budgets) {
            // the budgets of Eq. 5: one warp for up to 32 units, else the whole CTA
            const int cap = p.basis == TGVKV_BASIS_ALL ? p.N : p.N_v;
            const bool uniform = p.budget_stat == TGVKV_STAT_UNIFORM;
            if (units <= 32 && in_smem) {
                if (warp == 0)
                    tvb_budget_warp(lane < units ? us[lane] : 0.f, units, budget_total, cap, budgets,
                                    status, uniform, lane);
            } else {
                static_assert(sizeof(BudgetScratch) <= sizeof(s.k) / 2, "budget scratch in the K ring");
                tvb_budget_block(tvb_stat, units, budget_total, cap, budgets, status,
                                 *reinterpret_cast<BudgetScratch*>(reinterpret_cast<char*>(&s.k[0][0][0]) +
                                                                   sizeof(s.k) / 2),
                                 uniform);
            }
        }
        if (tid == 0) *exit_counter = 0u;
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

template <int D, int MODE>
cudaError_t launch_mode(const CUtensorMap& mq, const CUtensorMap& mk, const Problem& p, int n_items,
                        int n_two, const uint8_t* modality, const int32_t* text_pos, const float* w,
                        float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                        long long budget_total, int32_t* budgets, cudaStream_t stream) {
    static_assert(sizeof(PSmem<D>) + 1024 <= 227 * 1024, "shared memory of one CTA");
    const size_t smem = sizeof(PSmem<D>) + 1024;
    cudaError_t e = cudaFuncSetAttribute(score_tc_kernel<D, MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(score_tc_kernel<D, MODE>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    const int sms = sm_count();
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int grid = n_items < sms ? n_items : sms;
    // a programmatic dependent of the kernel before (it may begin while that one ends)
    return launch_dependent(score_tc_kernel<D, MODE>, dim3(grid), dim3(NTHREADS), smem, stream, mq, mk,
                            p, n_items, n_two, modality, text_pos, w, scores, tvb_stat,
                            reinterpret_cast<float*>(ws + lay.score_part),
                            reinterpret_cast<float*>(ws + lay.stat_part),
                            reinterpret_cast<float*>(ws + lay.stat_head),
                            reinterpret_cast<uint32_t*>(ws + lay.tickets),
                            reinterpret_cast<uint32_t*>(ws + lay.status), budget_total, budgets);
}

template <int D>
cudaError_t launch_tc(const Problem& p, const uint16_t* q, const uint16_t* k,
                      const uint8_t* modality, const int32_t* text_pos, const float* w,
                      float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                      long long budget_total, int32_t* budgets, cudaStream_t stream) {
    alignas(64) CUtensorMap mq, mk;
    if (!make_map(&mq, q, (uint64_t)p.L * p.H_q * p.n_win, D, 32) ||
        !make_map(&mk, k, (uint64_t)p.L * p.H_kv * p.N, D, BN))
        return cudaErrorInvalidValue;
    // the item shape: pairs of row tiles, or one row tile per head, or two
    // heads of at most 64 rows each packed into one row tile
    const int LH = p.L * p.H_kv;
    if (p.T >= 2)
        return launch_mode<D, MODE_PAIR>(mq, mk, p, LH * score_pairs(p), 0, modality, text_pos, w,
                                         scores, tvb_stat, ws, lay, budget_total, budgets, stream);
    if (2 * p.R <= BM) {
        // Two heads per item in whole rounds of the grid, one head per item for
        // the rest: the last round then spreads over up to twice as many CTAs
        // (1024 heads on 152 SMs: 3 rounds of two-head items, 112 one-head items).
        const int sms = sm_count();
        if (sms <= 0) return cudaErrorInvalidDevice;
        const int n_two = LH / 2 >= sms ? sms * ((LH / 2) / sms) : LH / 2;
        const int n_items = n_two + (LH - 2 * n_two);
        return launch_mode<D, MODE_PACKED>(mq, mk, p, n_items, n_two, modality, text_pos, w, scores,
                                           tvb_stat, ws, lay, budget_total, budgets, stream);
    }
    return launch_mode<D, MODE_SINGLE>(mq, mk, p, LH, 0, modality, text_pos, w, scores, tvb_stat, ws,
                                       lay, budget_total, budgets, stream);
}

}  // namespace

bool make_tile_map(CUtensorMap* map, const void* base, uint64_t rows, int d, uint32_t box_rows) {
    return make_map(map, base, rows, d, box_rows);
}

int device_sm_count() { return sm_count(); }

int score_launches(const Problem& p) { return p.R == 0 ? 0 : 1; }

cudaError_t launch_score(const Problem& p, const uint16_t* q, const uint16_t* k,
                         const uint8_t* modality, const int32_t* text_pos, const float* w,
                         float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                         long long budget_total, int32_t* budgets, cudaStream_t stream) {
    if (p.R == 0) {  // no query rows: no attention mass anywhere
        cudaError_t e = cudaSuccess;
        if (p.N_v > 0)
            e = cudaMemsetAsync(scores, 0, sizeof(float) * (size_t)p.L * p.H_kv * p.N_v, stream);
        const size_t units = p.head_budgets ? (size_t)p.L * p.H_kv : (size_t)p.L;
        if (e == cudaSuccess) e = cudaMemsetAsync(tvb_stat, 0, sizeof(float) * units, stream);
        return e;
    }
    if (p.d == 64)
        return launch_tc<64>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, budget_total,
                             budgets, stream);
    return launch_tc<128>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, budget_total,
                          budgets, stream);
}

}  // namespace tgvkv
