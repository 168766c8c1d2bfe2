// TWR scores and TVB statistic on the 5th-generation tensor cores (tcgen05).
//
// One CTA owns up to 128 query rows of one (layer, KV head) -- the G query
// heads of the group stacked over the n_win text-query rows -- and streams the
// head's 128-key tiles twice, the two passes of Eq. 2 / Eq. 8:
//
//   pass A  S = Q K^T  (TMEM lane = query row).  Each row keeps an online
//           maximum m_i, normaliser Z_i and vision mass V_i over every visible
//           key (causal: key j <= position of row i).
//   pass B  S^T = K Q^T  (TMEM lane = key) for the tiles that hold vision keys.
//           Each key j sums, over the rows, c_i 2^(x_ij - m_i) with
//           c_i = w_i / (G Z_i) -- the text-weighted column sum of Eq. 8 with
//           the GQA mean folded in.  The factor is folded into the exponent,
//           2^(x_ij - m'_i) with m'_i = m_i - log2 c_i, so a term costs one FFMA,
//           one EX2 and one FADD, and the column sum needs no cross-lane
//           reduction.
//
// Roles (320 threads): warp 0 issues TMA loads (Q once, then every K tile of
// both passes through a 2-stage ring); warp 1 owns the tensor memory (two
// 128-column fp32 accumulators) and one of its lanes issues the MMAs; warps
// 2-9 read the accumulators (tcgen05.ld) and do the softmax arithmetic, two
// warps per TMEM lane quarter, each taking half of a tile's columns.  Every
// wait is bounded (mbarrier try_wait with a 1 s limit); a timeout sets
// TGVKV_STATUS_TIMEOUT and the CTA unwinds.
//
// Query rows are spread evenly over the four lane quarters (row q*rpg + i ->
// lane 32q + i) so that all softmax warps share the work when a tile holds
// fewer than 128 rows.  Several row tiles per KV head (grouped-query layouts)
// write partial score rows; the last CTA of a head adds them in tile order and
// the last head of a layer adds the TV masses in head order, so results do not
// depend on the schedule.
#include <cudaTypedefs.h>
#include <limits.h>
#include <math.h>

#include "common.cuh"
#include "launch.h"
#include "tc05.cuh"

namespace tgvkv {
namespace {

constexpr int BM = 128;          // query rows per CTA = TMEM lanes
constexpr int BN = 128;          // keys per tile
constexpr int STAGES = 2;        // K tiles in flight per CTA
constexpr int NSOFT = 256;       // softmax threads (warps 2..9)
constexpr int NTHREADS = 64 + NSOFT;
constexpr int TMEM_COLS = 256;   // two 128-column accumulators
constexpr int MAXT = kMaxN / BN;
constexpr uint32_t IDESC = tc::idesc_bf16(128, 128);

template <int D>
struct TcSmem {
    uint16_t q[D / 64][BM * 64];            // Q tile, one 128-byte-swizzled half per 64 dims
    uint16_t k[STAGES][D / 64][BN * 64];    // K ring
    uint64_t full[STAGES], empty[STAGES], s_full[2], s_empty[2], q_full, mma_done;
    uint64_t pb_full[4][2], pb_empty[4][2]; // pass-B half-column hand-off per lane quarter
    uint32_t vmask[MAXT][4];                // vision bit of each key of each tile
    int vis_before[MAXT + 1];               // vision keys before each tile
    alignas(16) int row_pos[BM];            // per TMEM lane: position of its row, -1 = none
    float row_w[BM];
    alignas(16) float row_mp[BM];           // per TMEM lane: m_i - log2 c_i (+inf = no row)
    float row_mass[BM];                     // per TMEM lane: V_i / Z_i
    float part_m[BM], part_z[BM], part_v[BM];
    float pbuf[2][BM];
    uint32_t tmem_base;
    int max_pos, min_pos, abort_flag, never, is_last;
    float tile_mass;
};

template <int D>
constexpr size_t tc_smem_bytes() {
    // +1024 to align the tiles; at least 80 KB so that no more than two CTAs
    // share an SM (two 256-column accumulators fill its tensor memory)
    return sizeof(TcSmem<D>) + 1024 > 80 * 1024 ? sizeof(TcSmem<D>) + 1024 : 80 * 1024;
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
// MASKED), and the part of it over the vision keys flagged in vm.
template <bool MASKED>
__device__ __forceinline__ void exp_word(const float (&x)[32], float sl2, float nm, int lim,
                                         uint32_t vm, float& z, float& v) {
    float z0 = 0.f, z1 = 0.f, z2 = 0.f, z3 = 0.f;
    if (vm == 0u || vm == 0xFFFFFFFFu) {
#pragma unroll
        for (int c = 0; c < 32; c += 4) {
            float e0 = fast_exp2(fmaf(x[c], sl2, nm)), e1 = fast_exp2(fmaf(x[c + 1], sl2, nm));
            float e2 = fast_exp2(fmaf(x[c + 2], sl2, nm)), e3 = fast_exp2(fmaf(x[c + 3], sl2, nm));
            if (MASKED) {
                if (c > lim) e0 = 0.f;
                if (c + 1 > lim) e1 = 0.f;
                if (c + 2 > lim) e2 = 0.f;
                if (c + 3 > lim) e3 = 0.f;
            }
            z0 += e0; z1 += e1; z2 += e2; z3 += e3;
        }
        const float zs = (z0 + z1) + (z2 + z3);
        z += zs;
        if (vm) v += zs;
    } else {
        float v0 = 0.f, v1 = 0.f;
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
            float e0 = fast_exp2(fmaf(x[c], sl2, nm)), e1 = fast_exp2(fmaf(x[c + 1], sl2, nm));
            if (MASKED) {
                if (c > lim) e0 = 0.f;
                if (c + 1 > lim) e1 = 0.f;
            }
            z0 += e0; z1 += e1;
            v0 += ((vm >> c) & 1u) ? e0 : 0.f;
            v1 += ((vm >> (c + 1)) & 1u) ? e1 : 0.f;
        }
        z += z0 + z1;
        v += v0 + v1;
    }
}

// Sum over the valid rows of one 32-row group of 2^(y_i sl2 - mp_i), with the
// causal mask j <= pos_i unless every row sees key j.
__device__ __forceinline__ float colsum_group(const float (&y)[32], const float* mp,
                                              const int* pos, float sl2, int rpg, int j,
                                              bool all_vis) {
    float a0 = 0.f, a1 = 0.f;
#pragma unroll
    for (int i = 0; i < 32; i += 4) {
        if (i < rpg) {
            const float4 m4 = *reinterpret_cast<const float4*>(mp + i);
            float e0 = fast_exp2(fmaf(y[i], sl2, -m4.x));
            float e1 = fast_exp2(fmaf(y[i + 1], sl2, -m4.y));
            float e2 = fast_exp2(fmaf(y[i + 2], sl2, -m4.z));
            float e3 = fast_exp2(fmaf(y[i + 3], sl2, -m4.w));
            if (!all_vis) {
                const int4 p4 = *reinterpret_cast<const int4*>(pos + i);
                if (j > p4.x) e0 = 0.f;
                if (j > p4.y) e1 = 0.f;
                if (j > p4.z) e2 = 0.f;
                if (j > p4.w) e3 = 0.f;
            }
            a0 += e0 + e1;
            a1 += e2 + e3;
        }
    }
    return a0 + a1;
}

template <int D>
__global__ void __launch_bounds__(NTHREADS, 2)
score_tc_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                Problem p, const uint8_t* __restrict__ modality,
                const int32_t* __restrict__ text_pos, const float* __restrict__ w,
                float* __restrict__ scores, float* __restrict__ tvb_stat,
                float* __restrict__ score_part, float* __restrict__ stat_part,
                float* __restrict__ stat_head, uint32_t* __restrict__ tickets,
                uint32_t* __restrict__ status) {
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    TcSmem<D>& s = *reinterpret_cast<TcSmem<D>*>(smem_raw + (((raw + 1023u) & ~1023u) - raw));
    constexpr uint32_t TILE_BYTES = (D / 64) * BN * 128;   // one K tile = one Q tile

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int lh = blockIdx.y, l = lh / p.H_kv, g = lh % p.H_kv, t = blockIdx.x;
    const int row0 = t * BM;
    const int rows_t = min(BM, p.R - row0);
    const int rpg = (rows_t + 3) >> 2;          // rows per TMEM lane quarter
    const float sl2 = p.scale_log2;

    // ------------------------------------------------------------ prologue
    if (blockIdx.x == 0 && blockIdx.y == 0) {
        for (int i = tid; i < p.n_win; i += NTHREADS) {
            const int pi = text_pos[i];
            if (pi < 0 || pi >= p.N || (i > 0 && text_pos[i - 1] >= pi))
                raise_status(status, TGVKV_STATUS_TEXT_POS);
        }
    }
    if (tid == 0) {
        s.max_pos = -1;
        s.min_pos = INT_MAX;
        s.abort_flag = 0;
        s.never = 0;
        for (int i = 0; i < STAGES; ++i) {
            tc::mbar_init(&s.full[i], 1);
            tc::mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&s.s_full[i], 1);
            tc::mbar_init(&s.s_empty[i], NSOFT);
        }
        for (int qq = 0; qq < 4; ++qq)
            for (int i = 0; i < 2; ++i) {
                tc::mbar_init(&s.pb_full[qq][i], 32);
                tc::mbar_init(&s.pb_empty[qq][i], 32);
            }
        tc::mbar_init(&s.q_full, 1);
        tc::mbar_init(&s.mma_done, 1);
        tc::fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&s.tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    if (tid < BM) {
        const int qg = tid >> 5, i = tid & 31, rr = qg * rpg + i;
        int pos = -1;
        float wr = 0.f;
        if (i < rpg && rr < rows_t) {
            const int wi = (row0 + rr) % p.n_win;
            pos = text_pos[wi];
            if (pos < 0 || pos >= p.N) pos = -1;
            wr = w[(long long)l * p.w_stride + wi];
            if (!(wr >= 0.f) || isinf(wr)) {
                raise_status(status, TGVKV_STATUS_WEIGHT);
                wr = 0.f;
            }
        }
        s.row_pos[tid] = pos;
        s.row_w[tid] = wr;
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
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    if (tid < BM && s.row_pos[tid] >= 0) {
        atomicMax(&s.max_pos, s.row_pos[tid]);
        atomicMin(&s.min_pos, s.row_pos[tid]);
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
            if (blockIdx.x == 0 && blockIdx.y == 0 && total != p.N_v)
                raise_status(status, TGVKV_STATUS_VISION_COUNT);
        }
    }
    __syncthreads();
    const uint32_t tmem = s.tmem_base;
    const int n_tiles = (s.max_pos + BN) / BN;   // tiles holding keys 0..max_pos
    volatile int* abort_flag = &s.abort_flag;

    // ------------------------------------------------------------ TMA producer
    if (warp == 0 && lane == 0) {
        tc::tma_prefetch_desc(&tmap_q);
        tc::tma_prefetch_desc(&tmap_k);
        const int qy = (l * p.H_q + g * p.G) * p.n_win + row0;
        tc::mbar_arrive_expect_tx(&s.q_full, TILE_BYTES);
#pragma unroll
        for (int qg = 0; qg < 4; ++qg)
#pragma unroll
            for (int h = 0; h < D / 64; ++h)
                tc::tma_load_2d(&s.q[h][qg * 32 * 64], &tmap_q, h * 64, qy + qg * rpg, &s.q_full);
        int it = 0;
        bool ok = true;
        auto issue = [&](int kt) {
            const int stage = it % STAGES;
            if (!tc::mbar_wait(&s.empty[stage], ((it / STAGES) & 1) ^ 1, abort_flag)) {
                ok = false;
                return;
            }
            tc::mbar_arrive_expect_tx(&s.full[stage], TILE_BYTES);
#pragma unroll
            for (int h = 0; h < D / 64; ++h)
                tc::tma_load_2d(&s.k[stage][h][0], &tmap_k, h * 64, lh * p.N + kt * BN, &s.full[stage]);
            ++it;
        };
        for (int kt = 0; ok && kt < n_tiles; ++kt) issue(kt);
        for (int kt = next_vis_tile(s.vis_before, 0, n_tiles); ok && kt < n_tiles;
             kt = next_vis_tile(s.vis_before, kt + 1, n_tiles))
            issue(kt);
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every copy this CTA issued has landed before it may exit
        tc::mbar_wait(&s.q_full, 0, &s.never);
        for (int i = max(0, it - STAGES); i < it; ++i)
            tc::mbar_wait(&s.full[i % STAGES], (i / STAGES) & 1, &s.never);
    }

    // ------------------------------------------------------------ MMA issuer
    if (warp == 1 && lane == 0) {
        bool ok = tc::mbar_wait(&s.q_full, 0, abort_flag);
        int it = 0, st = 0;
        const uint32_t qa = smem_u32(&s.q[0][0]);
        auto mma_tile = [&](bool transposed) {
            const int stage = it % STAGES, buf = st & 1;
            if (!tc::mbar_wait(&s.full[stage], (it / STAGES) & 1, abort_flag) ||
                !tc::mbar_wait(&s.s_empty[buf], ((st >> 1) & 1) ^ 1, abort_flag)) {
                ok = false;
                return;
            }
            tc::fence_after_sync();
            const uint32_t ka = smem_u32(&s.k[stage][0][0]);
            const uint32_t d_tmem = tmem + (uint32_t)(buf * BN);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                const uint32_t off = (uint32_t)((kk >> 2) * (BM * 64 * 2) + (kk & 3) * 32);
                const uint64_t qd = tc::sdesc_k_sw128(qa + off);
                const uint64_t kd = tc::sdesc_k_sw128(ka + off);
                tc::mma_bf16(d_tmem, transposed ? kd : qd, transposed ? qd : kd, IDESC, kk > 0);
            }
            tc::mma_commit(&s.empty[stage]);
            tc::mma_commit(&s.s_full[buf]);
            ++it;
            ++st;
        };
        if (ok)
            for (int kt = 0; ok && kt < n_tiles; ++kt) mma_tile(false);
        for (int kt = next_vis_tile(s.vis_before, 0, n_tiles); ok && kt < n_tiles;
             kt = next_vis_tile(s.vis_before, kt + 1, n_tiles))
            mma_tile(true);
        if (!ok) {
            s.abort_flag = 1;
            raise_status(status, TGVKV_STATUS_TIMEOUT);
        }
        // every MMA this CTA issued has finished before TMEM is released
        tc::mma_commit(&s.mma_done);
        tc::mbar_wait(&s.mma_done, 0, &s.never);
    }

    // ------------------------------------------------------------ softmax warps
    if (warp >= 2) {
        const int quarter = warp & 3;
        const int hf = (warp - 2) >> 2;                     // which 64 columns of a tile
        const int ln = quarter * 32 + lane;                 // this thread's TMEM lane
        const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(hf * 64);
        const int my_pos = s.row_pos[ln];
        float m = -INFINITY, z = 0.f, v = 0.f;
        int st = 0;
        bool ok = true;

        // ---- pass A: row statistics over this thread's half of every tile
        for (int kt = 0; ok && kt < n_tiles; ++kt) {
            const int buf = st & 1;
            if (!tc::mbar_wait(&s.s_full[buf], (st >> 1) & 1, abort_flag)) {
                ok = false;
                s.abort_flag = 1;
                break;
            }
            tc::fence_after_sync();
            float x0[32], x1[32];
            __syncwarp();
            tc::tmem_ld32(tl + (uint32_t)(buf * BN), x0);
            tc::tmem_ld32(tl + (uint32_t)(buf * BN + 32), x1);
            tc::tmem_wait_ld();
            tc::fence_before_sync();
            tc::mbar_arrive(&s.s_empty[buf]);
            const int lim = my_pos - (kt * BN + hf * 64);   // columns 0..lim of this half visible
            if (lim >= 0) {
                const uint32_t vm0 = s.vmask[kt][hf * 2], vm1 = s.vmask[kt][hf * 2 + 1];
                if (lim >= 63) {
                    const float m_new = fmaxf(m, fmaxf(max32(x0), max32(x1)) * sl2);
                    const float alpha = fast_exp2(m - m_new);
                    z *= alpha;
                    v *= alpha;
                    exp_word<false>(x0, sl2, -m_new, 63, vm0, z, v);
                    exp_word<false>(x1, sl2, -m_new, 63, vm1, z, v);
                    m = m_new;
                } else {
                    const float m_new =
                        fmaxf(m, fmaxf(max32_masked(x0, lim), max32_masked(x1, lim - 32)) * sl2);
                    const float alpha = fast_exp2(m - m_new);
                    z *= alpha;
                    v *= alpha;
                    exp_word<true>(x0, sl2, -m_new, lim, vm0, z, v);
                    exp_word<true>(x1, sl2, -m_new, lim - 32, vm1, z, v);
                    m = m_new;
                }
            }
            ++st;
        }
        // ---- combine the two halves of each row
        if (hf == 1) {
            s.part_m[ln] = m;
            s.part_z[ln] = z;
            s.part_v[ln] = v;
        }
        tc::named_bar_sync(1, NSOFT);
        if (hf == 0) {
            const float m1 = s.part_m[ln];
            const float mt = fmaxf(m, m1);
            float zt = 0.f, vt = 0.f;
            if (mt != -INFINITY) {
                const float a0 = fast_exp2(m - mt), a1 = fast_exp2(m1 - mt);
                zt = z * a0 + s.part_z[ln] * a1;
                vt = v * a0 + s.part_v[ln] * a1;
            }
            const bool valid = my_pos >= 0 && zt > 0.f;
            // rows without attention get m' = +inf: every term 2^-inf = 0
            s.row_mp[ln] = valid ? mt - fast_log2(s.row_w[ln] / ((float)p.G * zt)) : INFINITY;
            s.row_mass[ln] = valid ? vt / zt : 0.f;
        }
        tc::named_bar_sync(1, NSOFT);
        if (tid == 64) {
            float a = 0.f;
            for (int r = 0; r < BM; ++r) a += s.row_mass[r];
            s.tile_mass = a;
        }

        // ---- pass B: text-weighted column sums, one key per thread
        float* out = (p.T == 1) ? scores + (size_t)lh * p.N_v
                                : score_part + ((size_t)lh * p.T + t) * p.N_v;
        const float* mp = s.row_mp + hf * 64;
        const int* rp = s.row_pos + hf * 64;
        int u = 0;                                          // pass-B tile count
        for (int kt = next_vis_tile(s.vis_before, 0, n_tiles); ok && kt < n_tiles;
             kt = next_vis_tile(s.vis_before, kt + 1, n_tiles)) {
            const int buf = st & 1;
            if (!tc::mbar_wait(&s.s_full[buf], (st >> 1) & 1, abort_flag)) {
                ok = false;
                s.abort_flag = 1;
                break;
            }
            tc::fence_after_sync();
            float y0[32], y1[32];
            __syncwarp();
            tc::tmem_ld32(tl + (uint32_t)(buf * BN), y0);
            tc::tmem_ld32(tl + (uint32_t)(buf * BN + 32), y1);
            tc::tmem_wait_ld();
            tc::fence_before_sync();
            tc::mbar_arrive(&s.s_empty[buf]);
            const int j = kt * BN + ln;                     // this thread's key
            const bool all_vis = kt * BN + BN - 1 <= s.min_pos;
            float acc = colsum_group(y0, mp, rp, sl2, rpg, j, all_vis) +
                        colsum_group(y1, mp + 32, rp + 32, sl2, rpg, j, all_vis);
            // hand the second half's sum to the first half's thread of this key
            const int b2 = u & 1;
            const uint32_t ph = (u >> 1) & 1;
            if (hf == 1) {
                if (!tc::mbar_wait(&s.pb_empty[quarter][b2], ph ^ 1, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                    break;
                }
                s.pbuf[b2][ln] = acc;
                tc::mbar_arrive(&s.pb_full[quarter][b2]);
            } else {
                if (!tc::mbar_wait(&s.pb_full[quarter][b2], ph, abort_flag)) {
                    ok = false;
                    s.abort_flag = 1;
                    break;
                }
                acc += s.pbuf[b2][ln];
                tc::mbar_arrive(&s.pb_empty[quarter][b2]);
                const uint32_t word = s.vmask[kt][quarter];
                if (j < p.N && ((word >> lane) & 1u)) {
                    int vr = s.vis_before[kt] + __popc(word & ((1u << lane) - 1u));
                    for (int q2 = 0; q2 < quarter; ++q2) vr += __popc(s.vmask[kt][q2]);
                    if (vr < p.N_v) out[vr] = acc;
                }
            }
            ++st;
            ++u;
        }
        if (!ok) raise_status(status, TGVKV_STATUS_TIMEOUT);
        // vision keys after every query row of this tile get no attention
        for (int vv = s.vis_before[n_tiles] + (tid - 64); vv < p.N_v; vv += NSOFT) out[vv] = 0.f;
    }

    // ------------------------------------------------------------ teardown
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, TMEM_COLS);
    }

    // ------------------------------------------------------------ reductions
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        int last = 1;
        if (p.T == 1) {
            stat_head[lh] = s.tile_mass;
        } else {
            stat_part[(size_t)lh * p.T + t] = s.tile_mass;
            __threadfence();
            const unsigned old = atomicAdd(&tickets[lh], 1u);
            last = (old == (unsigned)(p.T - 1));
        }
        s.is_last = last;
    }
    __syncthreads();
    if (!s.is_last) return;
    __threadfence();
    if (p.T > 1) {
        for (int vv = tid; vv < p.N_v; vv += NTHREADS) {
            float a = 0.f;
            for (int tt = 0; tt < p.T; ++tt) a += __ldcg(&score_part[((size_t)lh * p.T + tt) * p.N_v + vv]);
            scores[(size_t)lh * p.N_v + vv] = a;
        }
        if (tid == 0) {
            float a = 0.f;
            for (int tt = 0; tt < p.T; ++tt) a += __ldcg(&stat_part[(size_t)lh * p.T + tt]);
            stat_head[lh] = a;
            tickets[lh] = 0u;
        }
    }
    if (tid == 0) {
        __threadfence();
        const unsigned old = atomicAdd(&tickets[p.L * p.H_kv + l], 1u);
        if (old == (unsigned)(p.H_kv - 1)) {
            __threadfence();
            float S = 0.f;
            for (int gg = 0; gg < p.H_kv; ++gg) S += __ldcg(&stat_head[(size_t)l * p.H_kv + gg]);
            tvb_stat[l] = S;
            tickets[p.L * p.H_kv + l] = 0u;
        }
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

template <int D>
cudaError_t launch_tc(const Problem& p, const uint16_t* q, const uint16_t* k,
                      const uint8_t* modality, const int32_t* text_pos, const float* w,
                      float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                      cudaStream_t stream) {
    alignas(64) CUtensorMap mq, mk;
    if (!make_map(&mq, q, (uint64_t)p.L * p.H_q * p.n_win, D, 32) ||
        !make_map(&mk, k, (uint64_t)p.L * p.H_kv * p.N, D, BN))
        return cudaErrorInvalidValue;
    const size_t smem = tc_smem_bytes<D>();
    cudaError_t e = cudaFuncSetAttribute(score_tc_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(score_tc_kernel<D>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    dim3 grid(p.T, p.L * p.H_kv);
    score_tc_kernel<D><<<grid, NTHREADS, smem, stream>>>(
        mq, mk, p, modality, text_pos, w, scores, tvb_stat,
        reinterpret_cast<float*>(ws + lay.score_part), reinterpret_cast<float*>(ws + lay.stat_part),
        reinterpret_cast<float*>(ws + lay.stat_head), reinterpret_cast<uint32_t*>(ws + lay.tickets),
        reinterpret_cast<uint32_t*>(ws + lay.status));
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score_tc(const Problem& p, const uint16_t* q, const uint16_t* k,
                            const uint8_t* modality, const int32_t* text_pos, const float* w,
                            float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                            cudaStream_t stream) {
    if (p.d == 64)
        return launch_tc<64>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
    return launch_tc<128>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
}

}  // namespace tgvkv
