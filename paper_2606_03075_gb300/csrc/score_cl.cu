// TWR scores and TVB statistic for heads whose query rows fit one 128-row
// tile (G * n_win <= 128), with each head's keys split over the CTAs of a
// thread-block cluster, and pass B computed from terms kept in tensor memory.
//
// Work item = one (layer, KV head).  CTA r of a cluster of C CTAs owns the
// key slice [r Kc, (r+1) Kc), Kc <= 512, of every item its cluster takes
// (items cid, cid + clusters, ...).  The slice's keys stream once through a
// ring of shared-memory tiles (TMA, 32-key boxes); S = Q K^T of each
// 128-key tile lands in its own 128 columns of TMEM (TMEM lane = query row),
// so one item's logits fill at most the 512 columns.  Then:
//
//   pass A  per row the vision mass and normaliser over the slice's visible
//           keys (Eq. 2 rows, the Eq. 6 slice, Eq. 5 numerator), taking the
//           terms e_ij = 2^(x_ij - r_i) against a reference r_i set by the
//           row's first word (moved up only when a word's terms would grow
//           large), and writing e_ij back over the logits in TMEM (0 for keys
//           the row does not see).
//   merge   the CTA's (r, Z, V) of every row is stored into every CTA of the
//           cluster (asynchronous distributed-shared-memory stores counted in
//           bytes on the receiver's mbarrier); each CTA adds the C partials in
//           rank order, so all CTAs hold the same row statistics (m, Z, V).
//   pass B  Eq. 8 with the GQA mean: per key j the sum over rows of
//           a_i e_ij, a_i = w_i 2^(r_i - m_i) / (G Z_i), read back from TMEM:
//           one multiply per term and a 32-lane transpose-reduce per 32x32
//           block, no second product and no second exponential.
//
// K is read from HBM once; a tile's shared-memory slot is free as soon as its
// product is done, so the next item's tiles stream in while this item merges.
// The MMA of the next item's tile t waits only for pass B to have read TMEM
// tile t.
//
// Roles (576 threads): warp 0 issues the TMA loads; warp 1 owns the TMEM and
// its lane 0 issues the products; warps 2..17 run both passes, four per TMEM
// lane quarter, warp (quarter q, chunk c) owning columns [32c, 32c + 32) of
// every tile for the quarter's rows.  Sums run in a fixed order, so results
// do not depend on the schedule.  Every wait is bounded; a timeout sets
// TGVKV_STATUS_TIMEOUT and the CTA unwinds without waiting again.
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

constexpr int KT = 128;                 // keys per tile
constexpr int NSW = 16;                 // softmax warps
constexpr int NSOFT = NSW * 32;
constexpr int NTHREADS = (NSW + 2) * 32;
constexpr int MAXC = 8;                 // CTAs per cluster (portable limit)
constexpr int MAXT = 4;                 // tiles per CTA slice: 4 x 128 TMEM columns
constexpr int MAXNS = 8;                // K ring slots
constexpr int ROWS = 128;               // TMEM lanes
constexpr int TMEM_COLS = 512;
constexpr int D = 128;                  // head dimension of this kernel
constexpr float kRefSlack = 8.f;        // a word whose terms sum above 32 * 2^this is redone
constexpr uint32_t kMinSmem = 160u * 1024u;

// Fixed-size part of the shared memory (after the Q slots, the K ring and the
// merge buffers, whose sizes depend on the problem).
struct ClMisc {
    uint64_t q_full[2], q_empty[2];
    uint64_t k_full[MAXNS], k_empty[MAXNS];
    uint64_t t_full[MAXT], t_free[MAXT];    // TMEM tile written / read by pass B
    uint64_t xch_bar[2];
    uint64_t mma_done;
    float part[3][4][ROWS];                 // pass-A partials: [r, Z, V][warp of the quarter][row]
    float row_m[ROWS], row_c[ROWS];         // merged maximum m_i and w_i / (G Z_i) (0: no row)
    alignas(16) int row_pos[ROWS];          // position of each row, -1 = none
    float red[4][MAXT][KT];                 // pass-B sums over each quarter's rows
    float tmass[4];                         // TV mass per quarter
    uint32_t vmask[MAXT][4];                // vision keys of the slice, per 32-key word
    int vq[MAXT][4];                        // vision rank of each word's first key
    uint32_t tmem_base;
    int abort_flag, never, cta_last, vis_before_slice;
};

// Shared-memory carve-up (byte offsets from the 1024-aligned base).
struct ClLayout {
    uint32_t q, rb;          // Q: 2 slots x 2 dim-halves x rb (rq rows x 128 B)
    uint32_t k;              // K ring: ns slots of 2 x 128 keys x 128 B
    uint32_t xch;            // float [2 parity][3][C][rq]: every CTA's (r, Z, V) per row
    uint32_t misc;
    uint32_t total;          // bytes from the base, plus 1024 of alignment slack
    int rq;                  // Q rows stored per slot (R rounded up to 32)
    int C, Kc, ns;           // CTAs per cluster, keys per CTA slice, K ring slots
};

constexpr uint32_t kSlotBytes = 2u * KT * 128u;

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, abort);
    return __all_sync(~0u, got);
}

// D = A B^T over K = 128 (8 steps of 16); a / b: descriptors of the first
// 64-dim half, a_half / b_half: 16-byte units to the second half.
__device__ __forceinline__ void mma_k128(uint32_t d_tmem, uint64_t a, uint32_t a_half, uint64_t b,
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

// One 32-key word of a row in pass A: columns 0..lim visible, vm flags the
// vision keys.  Turns x into e = 2^(x sl2 - r) (0 beyond lim) against the
// row's reference r and returns its sum (vs: the sum over the vision keys).
// MASKED: some column is beyond lim; MIXED: vm is neither all nor none.
template <bool MASKED, bool MIXED>
__device__ __forceinline__ float exp_word_ref(float (&x)[32], float sl2, float r, int lim, uint32_t vm,
                                              float& vs) {
    const float2 s2 = make_float2(sl2, sl2), n2 = make_float2(-r, -r);
    float2 za = make_float2(0.f, 0.f), zb = za, va = za;
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
        x[c] = e0.x;
        x[c + 1] = e0.y;
        x[c + 2] = e1.x;
        x[c + 3] = e1.y;
        za = add2(za, e0);
        zb = add2(zb, e1);
        if (MIXED) {
            va = add2(va, make_float2((vm >> c) & 1u ? e0.x : 0.f, (vm >> (c + 1)) & 1u ? e0.y : 0.f));
            va = add2(va, make_float2((vm >> (c + 2)) & 1u ? e1.x : 0.f, (vm >> (c + 3)) & 1u ? e1.y : 0.f));
        }
    }
    const float zs = (za.x + za.y) + (zb.x + zb.y);
    vs = MIXED ? va.x + va.y : (vm ? zs : 0.f);
    return zs;
}

__device__ __forceinline__ float exp_word_any(float (&x)[32], float sl2, float r, int lim, uint32_t vm,
                                              float& vs) {
    const bool mixed = vm != 0u && vm != 0xFFFFFFFFu;
    if (lim >= 31)
        return mixed ? exp_word_ref<false, true>(x, sl2, r, lim, vm, vs)
                     : exp_word_ref<false, false>(x, sl2, r, lim, vm, vs);
    return mixed ? exp_word_ref<true, true>(x, sl2, r, lim, vm, vs)
                 : exp_word_ref<true, false>(x, sl2, r, lim, vm, vs);
}

// Pass A on the word at TMEM address ta (this warp's lanes): e written back,
// z and v accumulated.  The first visible word sets r to its maximum; later
// words keep r unless their sum passes 32 * 2^kRefSlack, i.e. some term may be
// large (or overflowed): then the logits are loaded again and the word is
// redone against its own maximum, which moves r up (z and v rescaled).  So
// every kept term is at most 32 * 2^kRefSlack and r never exceeds the row's
// maximum.  Returns with x holding the terms to store.
__device__ __forceinline__ void pass_a_word(float (&x)[32], uint32_t ta, float sl2, int lim, uint32_t vm,
                                            float& r, float& z, float& v) {
    const bool live = lim >= 0;   // the row sees a key of this word
    float zs = 0.f, vs = 0.f;
    bool redo = live && r == -INFINITY;
    if (live && !redo) {
        zs = exp_word_any(x, sl2, r, lim, vm, vs);
        redo = !(zs <= 32.f * (float)(1 << (int)kRefSlack));   // also true for inf and nan
    }
    // the TMEM load is warp-collective: every lane reloads its logits if any lane redoes
    if (__any_sync(~0u, redo)) {
        tc::tmem_ld32(ta, x);
        tc::tmem_wait_ld();
        if (live) {
            if (redo) {
                const float wm = (lim >= 31 ? max32(x) : max32_masked(x, lim)) * sl2;
                if (wm > r) {
                    const float a = fast_exp2(r - wm);   // r = -inf: a = 0 and z = v = 0 stay 0
                    z *= a;
                    v *= a;
                    r = wm;
                }
            }
            zs = exp_word_any(x, sl2, r, lim, vm, vs);   // unchanged r: the same terms again
        }
    }
    if (!live) {
#pragma unroll
        for (int c = 0; c < 32; ++c) x[c] = 0.f;
    }
    z += zs;
    v += vs;
}

// Sum over the warp's 32 lanes of v[k] for every k: afterwards lane L holds
// the sum for k = L (recursive halving, a fixed order).
__device__ __forceinline__ float transpose_reduce32(float (&v)[32], int lane) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const bool hi = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < o; ++i) {
            const float send = hi ? v[i] : v[i + o];
            const float keep = hi ? v[i + o] : v[i];
            v[i] = keep + __shfl_xor_sync(~0u, send, o);
        }
    }
    return v[0];
}

__global__ void __launch_bounds__(NTHREADS, 1)
score_cl_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                Problem p, ClLayout lay, int n_items, const uint8_t* __restrict__ modality,
                const int32_t* __restrict__ text_pos, const float* __restrict__ w,
                float* __restrict__ scores, float* __restrict__ tvb_stat,
                float* __restrict__ stat_head, uint32_t* __restrict__ exit_counter,
                uint32_t* __restrict__ status, long long budget_total, int32_t* __restrict__ budgets) {
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    unsigned char* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t sbase = smem_u32(base);
    ClMisc& s = *reinterpret_cast<ClMisc*>(base + lay.misc);
    float* xch = reinterpret_cast<float*>(base + lay.xch);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int C = lay.C, ns = lay.ns;
    const int rank = (int)tc::cluster_ctarank();
    const int cid = (int)tc::cluster_id_x(), ncl = (int)tc::cluster_count_x();
    const float sl2 = p.scale_log2;
    const int k0 = rank * lay.Kc;
    const int k1 = min(p.N, k0 + lay.Kc);
    const int nt = k1 > k0 ? (k1 - k0 + KT - 1) / KT : 0;   // tiles of this CTA's slice
    const int rq = lay.rq;
    const int nq = (p.R + 31) / 32;                         // lane quarters holding rows

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
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&s.q_full[i], 1);
            tc::mbar_init(&s.q_empty[i], 1);
            tc::mbar_init(&s.xch_bar[i], 1);        // this CTA's expect; the rows arrive as bytes
        }
        for (int i = 0; i < MAXNS; ++i) {
            tc::mbar_init(&s.k_full[i], 1);
            tc::mbar_init(&s.k_empty[i], 1);
        }
        for (int t = 0; t < MAXT; ++t) {
            tc::mbar_init(&s.t_full[t], 1);
            tc::mbar_init(&s.t_free[t], NSW);       // every softmax warp has read the tile
        }
        tc::mbar_init(&s.mma_done, 1);
        tc::fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&s.tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    // vision keys before this slice (block-wide count), rows, and per-word masks
    if (tid == 0) s.vis_before_slice = 0;
    if (tid < 4) s.tmass[tid] = 0.f;
    for (int r = tid; r < ROWS; r += NTHREADS) {
        int pos = -1;
        if (r < p.R) {
            pos = text_pos[r % p.n_win];
            if (pos < 0 || pos >= p.N) pos = -1;
        }
        s.row_pos[r] = pos;
    }
    __syncthreads();
    {
        int c = 0;
        for (int j = tid; j < k0; j += NTHREADS) c += modality[j] != 0;
        c = __reduce_add_sync(~0u, c);
        if (lane == 0 && c) atomicAdd(&s.vis_before_slice, c);
    }
    __syncthreads();
    if (warp == 0) {
        // masks of the slice's words (keys >= k1 belong to the next CTA), and
        // the vision rank of each word's first key
        int run = s.vis_before_slice;
        for (int t = 0; t < nt; ++t) {
#pragma unroll
            for (int wd = 0; wd < 4; ++wd) {
                const int j = k0 + t * KT + wd * 32 + lane;
                const unsigned m = __ballot_sync(~0u, j < k1 && modality[j] != 0);
                if (lane == 0) {
                    s.vmask[t][wd] = m;
                    s.vq[t][wd] = run;
                }
                run += __popc(m);
            }
        }
        // the last slice ends at N: its count is the head's vision count
        if (lane == 0 && k1 == p.N && run != p.N_v) raise_status(status, TGVKV_STATUS_VISION_COUNT);
    }
    // the largest row position
    int maxpos = -1;
    for (int r = 0; r < ROWS; ++r) maxpos = max(maxpos, s.row_pos[r]);
    __syncthreads();
    // tiles with a key some row sees (the others' vision scores are 0)
    int nA = 0;
    while (nA < nt && k0 + nA * KT <= maxpos) ++nA;
    int zv0 = 0, zv1 = 0;
    if (nA < nt) {
        zv0 = s.vq[nA][0];
        zv1 = s.vq[nt - 1][3] + __popc(s.vmask[nt - 1][3]);
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::cluster_sync();   // every CTA's barriers are initialised before any remote access
    tc::fence_after_sync();
    const uint32_t tmem = s.tmem_base;
    volatile int* abort_flag = &s.abort_flag;

    // ------------------------------------------------------------ producer
    if (warp == 0 && lane == 0) {
        tc::tma_prefetch_desc(&tmap_q);
        tc::tma_prefetch_desc(&tmap_k);
        bool ok = true;
        int n_items_mine = 0, g = 0;
        for (int n = 0; ok; ++n) {
            const int item = cid + n * ncl;
            if (item >= n_items) break;
            n_items_mine = n + 1;
            const int lh = item, l = lh / p.H_kv, gh = lh % p.H_kv;
            const int sq = n & 1;
            if (!tc::mbar_wait(&s.q_empty[sq], ((n >> 1) & 1) ^ 1, abort_flag)) {
                ok = false;
                break;
            }
            const int qrow0 = (l * p.H_q + gh * p.G) * p.n_win;
            tc::mbar_arrive_expect_tx(&s.q_full[sq], (uint32_t)(2 * rq * 128));
            for (int h = 0; h < 2; ++h)
                for (int b = 0; b < rq / 32; ++b)
                    tc::tma_load_2d(base + lay.q + (2 * sq + h) * lay.rb + b * 4096, &tmap_q, 64 * h,
                                    qrow0 + 32 * b, &s.q_full[sq]);
            for (int t = 0; t < nA; ++t, ++g) {
                const int slot = g % ns;
                if (!tc::mbar_wait(&s.k_empty[slot], ((g / ns) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const int keys = min(KT, k1 - (k0 + t * KT));
                const int boxes = (keys + 31) / 32;
                tc::mbar_arrive_expect_tx(&s.k_full[slot], (uint32_t)(2 * boxes * 4096));
                for (int h = 0; h < 2; ++h)
                    for (int b = 0; b < boxes; ++b)
                        tc::tma_load_2d(base + lay.k + slot * kSlotBytes + h * KT * 128 + b * 4096,
                                        &tmap_k, 64 * h, lh * p.N + k0 + t * KT + 32 * b, &s.k_full[slot]);
            }
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every copy this CTA issued has landed before it may exit
        for (int n = max(0, n_items_mine - 2); n < n_items_mine; ++n)
            tc::mbar_wait(&s.q_full[n & 1], (n >> 1) & 1, &s.never);
        for (int i = max(0, g - ns); i < g; ++i) tc::mbar_wait(&s.k_full[i % ns], (i / ns) & 1, &s.never);
    }

    // ------------------------------------------------------------ MMA issuer
    if (warp == 1 && lane == 0) {
        const uint32_t q_half = lay.rb / 16;
        constexpr uint32_t K_HALF = KT * 128 / 16;
        int g = 0;
        bool ok = true;
        for (int n = 0; ok; ++n) {
            const int item = cid + n * ncl;
            if (item >= n_items) break;
            const int sq = n & 1;
            if (!tc::mbar_wait(&s.q_full[sq], (n >> 1) & 1, abort_flag)) {
                ok = false;
                break;
            }
            const uint64_t qd = tc::sdesc_k_sw128(sbase + lay.q + 2 * sq * lay.rb);
            for (int t = 0; t < nA; ++t, ++g) {
                const int slot = g % ns;
                if (!tc::mbar_wait(&s.k_full[slot], (g / ns) & 1, abort_flag) ||
                    !tc::mbar_wait(&s.t_free[t], (n & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                const int ncols = (min(KT, k1 - (k0 + t * KT)) + 31) / 32 * 32;
                const uint64_t kd = tc::sdesc_k_sw128(sbase + lay.k + slot * kSlotBytes);
                mma_k128(tmem + (uint32_t)(t * KT), qd, q_half, kd, K_HALF, tc::idesc_bf16(128, ncols));
                tc::mma_commit(&s.k_empty[slot]);
                tc::mma_commit(&s.t_full[t]);
            }
            tc::mma_commit(&s.q_empty[sq]);
        }
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every MMA this CTA issued has finished before TMEM is released
        tc::mma_commit(&s.mma_done);
        tc::mbar_wait(&s.mma_done, 0, &s.never);
    }

    // ------------------------------------------------------------ both passes
    if (warp >= 2) {
        const int sid = tid - 64;
        const int quarter = warp & 3;
        const int wc = (warp - 2) >> 2;                 // this warp's 32-column chunk of a tile
        const int row = quarter * 32 + lane;
        const bool has_rows = quarter < nq;
        const uint32_t tq = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(32 * wc);
        const int my_pos = s.row_pos[row];
        const int last = min(my_pos, k1 - 1);
        bool ok = true;
        for (int n = 0;; ++n) {
            const int item = cid + n * ncl;
            if (item >= n_items) break;
            const int lh = item, l = lh / p.H_kv;
            const int par = n & 1;

            // the row's text weight, loaded now so that the merge does not wait for it
            float wr = 0.f;
            if (wc == 0 && has_rows && my_pos >= 0) wr = __ldg(&w[(long long)l * p.w_stride + row % p.n_win]);

            // ---- pass A: terms against the row's reference, written back to TMEM
            float r = -INFINITY, z = 0.f, v = 0.f;
            float rt[MAXT];
#pragma unroll
            for (int t = 0; t < MAXT; ++t) rt[t] = -INFINITY;
#pragma unroll
            for (int t = 0; t < MAXT; ++t) {
                if (t >= nA) break;
                if (ok && !warp_wait(&s.t_full[t], n & 1, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                }
                if (!ok || !has_rows) continue;
                tc::fence_after_sync();
                float x[32];
                tc::tmem_ld32(tq + (uint32_t)(t * KT), x);
                tc::tmem_wait_ld();
                const int ws = k0 + t * KT + 32 * wc;
                pass_a_word(x, tq + (uint32_t)(t * KT), sl2, last - ws, s.vmask[t][wc], r, z, v);
                rt[t] = r;
                tc::tmem_st32(tq + (uint32_t)(t * KT), x);
            }
            tc::tmem_wait_st();

            // ---- the CTA's partial of each row, then every CTA's, in rank order
            s.part[0][wc][row] = r;
            s.part[1][wc][row] = z;
            s.part[2][wc][row] = v;
            tc::named_bar_sync(1 + quarter, 128);
            if (wc == 0 && has_rows) {
                float mt = -INFINITY, zt = 0.f, vt = 0.f;
#pragma unroll
                for (int c = 0; c < 4; ++c) mt = fmaxf(mt, s.part[0][c][row]);
                if (mt != -INFINITY) {
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const float a = fast_exp2(s.part[0][c][row] - mt);
                        zt += s.part[1][c][row] * a;
                        vt += s.part[2][c][row] * a;
                    }
                }
                // this CTA expects the rows of every CTA (3 floats of each of rq rows);
                // a CTA that gave up neither expects nor publishes
                if (ok && quarter == 0 && lane == 0)
                    tc::mbar_arrive_expect_tx(&s.xch_bar[par], (uint32_t)(C * rq * 12));
                if (ok && row < rq) {
                    const uint32_t a0 =
                        sbase + lay.xch + (uint32_t)((((par * 3) * C + rank) * rq + row) * 4);
                    const uint32_t stride = (uint32_t)(C * rq * 4);
                    const uint32_t bar = smem_u32(&s.xch_bar[par]);
                    for (int q = 0; q < C; ++q) {
                        const uint32_t rb = tc::map_to_rank(bar, (uint32_t)q);
                        tc::st_async_f32(tc::map_to_rank(a0, (uint32_t)q), mt, rb);
                        tc::st_async_f32(tc::map_to_rank(a0 + stride, (uint32_t)q), zt, rb);
                        tc::st_async_f32(tc::map_to_rank(a0 + 2 * stride, (uint32_t)q), vt, rb);
                    }
                }
                if (ok && !tc::mbar_wait_cluster(&s.xch_bar[par], (n >> 1) & 1, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                }
                float M = -INFINITY, Z = 0.f, V = 0.f;
                if (ok && row < rq) {
                    const float* xm = xch + (size_t)(par * 3) * C * rq + row;
                    const float* xz = xm + (size_t)C * rq;
                    const float* xv = xz + (size_t)C * rq;
                    for (int q = 0; q < C; ++q) M = fmaxf(M, xm[(size_t)q * rq]);
                    if (M != -INFINITY) {
                        for (int q = 0; q < C; ++q) {
                            const float a = fast_exp2(xm[(size_t)q * rq] - M);
                            Z += xz[(size_t)q * rq] * a;
                            V += xv[(size_t)q * rq] * a;
                        }
                    }
                }
                if (my_pos >= 0 && (!(wr >= 0.f) || isinf(wr))) {
                    raise_status(status, TGVKV_STATUS_WEIGHT);
                    wr = 0.f;
                }
                const bool valid = my_pos >= 0 && Z > 0.f;
                s.row_m[row] = M;
                s.row_c[row] = valid ? wr / ((float)p.G * Z) : 0.f;
                float mass = valid ? V / Z : 0.f;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) mass += __shfl_xor_sync(~0u, mass, o);
                if (lane == 0) s.tmass[quarter] = mass;
            }
            tc::named_bar_sync(1 + quarter, 128);

            // ---- pass B: a_i e_ij summed over the quarter's rows, per key
            const float cr = s.row_c[row], mr = s.row_m[row];
#pragma unroll
            for (int t = 0; t < MAXT; ++t) {
                if (t >= nA) break;
                if (ok && has_rows) {
                    float e[32];
                    tc::tmem_ld32(tq + (uint32_t)(t * KT), e);
                    tc::tmem_wait_ld();
                    tc::fence_before_sync();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&s.t_free[t]);
                    // a = 0 for rows without attention, and for words the row never reached
                    const float a = (cr > 0.f && rt[t] != -INFINITY) ? cr * fast_exp2(rt[t] - mr) : 0.f;
#pragma unroll
                    for (int c = 0; c < 32; ++c) e[c] *= a;
                    s.red[quarter][t][32 * wc + lane] = transpose_reduce32(e, lane);
                } else if (ok) {
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&s.t_free[t]);
                }
            }
            tc::named_bar_sync(5, NSOFT);
            // ---- per key the quarters' sums in order; the vision keys' scores
            if (ok) {
                for (int kk = sid; kk < nA * KT; kk += NSOFT) {
                    const int t = kk / KT, col = kk % KT;
                    const uint32_t word = s.vmask[t][col >> 5];
                    if ((word >> (col & 31)) & 1u) {
                        float a = 0.f;
                        for (int q = 0; q < nq; ++q) a += s.red[q][t][col];
                        const int vr = s.vq[t][col >> 5] + __popc(word & ((1u << (col & 31)) - 1u));
                        if (vr < p.N_v) scores[(size_t)lh * p.N_v + vr] = a;
                    }
                }
                if (sid == 0 && rank == 0)
                    stat_head[lh] = (s.tmass[0] + s.tmass[1]) + (s.tmass[2] + s.tmass[3]);
            }
            for (int vv = zv0 + sid; vv < min(zv1, p.N_v); vv += NSOFT)
                scores[(size_t)lh * p.N_v + vv] = 0.f;
            // the sums and row values are read before the next item rewrites them
            tc::named_bar_sync(5, NSOFT);
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
    // no CTA leaves while another may still store into its shared memory
    tc::cluster_sync();
    // the last CTA to finish adds the per-head TV masses of each layer, in head order
    if (tid == 0) {
        __threadfence();
        s.cta_last = atomicAdd(exit_counter, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (s.cta_last) {
        __threadfence();
        if (p.head_budgets) {
            for (int lh = tid; lh < p.L * p.H_kv; lh += NTHREADS) tvb_stat[lh] = __ldcg(&stat_head[lh]);
        } else {
            for (int l = tid; l < p.L; l += NTHREADS) {
                float S = 0.f;
                for (int g = 0; g < p.H_kv; ++g) S += __ldcg(&stat_head[(size_t)l * p.H_kv + g]);
                tvb_stat[l] = S;
            }
        }
        if (budgets) {
            // the budgets of Eq. 5, with the now idle K ring as scratch
            __syncthreads();
            tvb_budget_block(tvb_stat, p.head_budgets ? p.L * p.H_kv : p.L, budget_total,
                             p.basis == TGVKV_BASIS_ALL ? p.N : p.N_v, budgets, status,
                             *reinterpret_cast<BudgetScratch*>(base + lay.k),
                             p.budget_stat == TGVKV_STAT_UNIFORM);
        }
        if (tid == 0) *exit_counter = 0u;
    }
}

// ---- host ---------------------------------------------------------------------
int max_smem_optin() {
    static int v[64] = {};
    static std::mutex mu;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!v[dev]) cudaDeviceGetAttribute(&v[dev], cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    return v[dev];
}

// The carve-up for C CTAs per cluster with the deepest K ring that fits (at
// least 2 slots); false if none fits or a slice exceeds the TMEM columns.
bool layout_for(const Problem& p, int C, ClLayout* out) {
    const int limit = max_smem_optin();
    if (limit <= 0) return false;
    ClLayout L{};
    L.C = C;
    L.rq = (p.R + 31) / 32 * 32;
    L.Kc = ((p.N + C - 1) / C + 31) / 32 * 32;
    if ((L.Kc + KT - 1) / KT > MAXT || L.rq > ROWS) return false;
    L.rb = (uint32_t)L.rq * 128u;
    L.q = 0;
    L.k = 4 * L.rb;
    for (int ns = MAXNS; ns >= 2; --ns) {
        L.ns = ns;
        uint32_t ring = (uint32_t)ns * kSlotBytes;
        if (ring < sizeof(BudgetScratch)) ring = sizeof(BudgetScratch);   // the last CTA's scratch
        // an MMA reads 128 rows of a Q slot (rq may be fewer): the K ring follows the Q slots
        L.xch = L.k + ring;
        L.misc = (L.xch + (uint32_t)(2 * 3 * C * L.rq * 4) + 15u) & ~15u;
        L.total = L.misc + (uint32_t)sizeof(ClMisc) + 1024u;
        // more than half of an SM's shared memory: one CTA per SM, so that no two
        // CTAs ever compete for the SM's 512 TMEM columns
        if (L.total < kMinSmem) L.total = kMinSmem;
        if (L.total <= (uint32_t)limit) {
            *out = L;
            return true;
        }
    }
    return false;
}

int max_clusters(const ClLayout& lay) {
    static int cache[64][MAXC + 1] = {};
    static std::mutex mu;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(mu);
    int& c = cache[dev][lay.C];
    if (c == 0) {
        if (cudaFuncSetAttribute(score_cl_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)lay.total) != cudaSuccess)
            return 0;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = lay.C;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(lay.C);
        cfg.blockDim = dim3(NTHREADS);
        cfg.dynamicSmemBytes = lay.total;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, score_cl_kernel, &cfg) != cudaSuccess) n = 0;
        c = n > 0 ? n : -1;
    }
    return c;
}

// The smallest cluster whose slices fit the TMEM columns and shared memory.
bool plan(const Problem& p, ClLayout* lay) {
    for (int C = 1; C <= MAXC; ++C)
        if (layout_for(p, C, lay)) return true;
    return false;
}

}  // namespace

bool score_cluster_eligible(const Problem& p) {
    if (p.d != D || p.T != 1 || p.R <= 64 || p.R > ROWS || p.keys_text || p.stats_given) return false;
    ClLayout lay;
    return plan(p, &lay);
}

cudaError_t launch_score_cluster(const Problem& p, const uint16_t* q, const uint16_t* k,
                                 const uint8_t* modality, const int32_t* text_pos, const float* w,
                                 float* scores, float* tvb_stat, char* ws, const WsLayout& wl,
                                 long long budget_total, int32_t* budgets, cudaStream_t stream) {
    ClLayout lay;
    if (!plan(p, &lay)) return cudaErrorInvalidConfiguration;
    alignas(64) CUtensorMap mq, mk;
    if (!make_tile_map(&mq, q, (uint64_t)p.L * p.H_q * p.n_win, D, 32) ||
        !make_tile_map(&mk, k, (uint64_t)p.L * p.H_kv * p.N, D, 32))
        return cudaErrorInvalidValue;
    const int ncl_max = max_clusters(lay);
    if (ncl_max <= 0) return cudaErrorInvalidConfiguration;
    const int n_items = p.L * p.H_kv;
    const int ncl = n_items < ncl_max ? n_items : ncl_max;
    cudaError_t e = cudaFuncSetAttribute(score_cl_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)lay.total);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = lay.C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(ncl * lay.C);
    cfg.blockDim = dim3(NTHREADS);
    cfg.dynamicSmemBytes = lay.total;
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    uint32_t* tickets = reinterpret_cast<uint32_t*>(ws + wl.tickets);
    uint32_t* exit_counter = tickets + (size_t)p.L * p.H_kv + 2;
    e = cudaLaunchKernelEx(&cfg, score_cl_kernel, mq, mk, p, lay, n_items, modality, text_pos, w,
                           scores, tvb_stat, reinterpret_cast<float*>(ws + wl.stat_head), exit_counter,
                           reinterpret_cast<uint32_t*>(ws + wl.status), budget_total, budgets);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace tgvkv
