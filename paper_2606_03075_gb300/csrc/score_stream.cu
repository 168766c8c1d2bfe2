// TWR scores and TVB statistic: streaming two-pass kernel (warp MMA).
//
// One CTA owns up to 128 query rows of one (layer, KV head): the G query heads
// of the group times the n_win text-query rows, stacked (row r = head
// r / n_win, window row r % n_win).  It streams the key tiles of the head
// twice:
//   pass A  logits x = scale * q k^T (Eq. 2) for every visible key, online
//           row maximum m_i, normaliser Z_i = sum_j 2^(x_ij - m_i) over all
//           visible keys and vision mass V_i over the vision keys;
//   pass B  the same logits for the tiles that hold vision keys; the text-
//           weighted probability c_i 2^(x_ij - m_i), c_i = w_i / (G Z_i), is
//           summed over the CTA's rows for every vision column (Eq. 8 with the
//           GQA mean folded into c_i).
// The K tiles of pass B were read moments before by pass A, so they come back
// from L2.  With several row tiles per head (grouped-query layouts) each CTA
// writes a partial score row; the last CTA of the head (completion counter)
// adds the partials in tile order, so the result does not depend on the
// schedule.  The TVB statistic S_l (Eq. 5, x = TV) is the sum of V_i / Z_i
// over rows, tiles and heads, reduced the same way.
#include <math.h>

#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int BM = 128;          // query rows per CTA
constexpr int BN = 64;           // keys per tile
constexpr int NWARP = 8;         // 16 rows per warp
constexpr int NTHREAD = NWARP * 32;
constexpr int MAX_TILES = kMaxN / BN;

template <int D>
struct StreamSmem {
    alignas(128) uint16_t q[BM * D];
    alignas(128) uint16_t k[2][BN * D];
    int vis_before[MAX_TILES + 1];  // vision keys before each key tile
    int vr[2][BN];                  // vision rank of each column of a tile, -1 = text
    float colsum[NWARP][BN];
    int pos[BM];
    float wrow[BM];
    float m[BM];     // row maximum of the base-2 logits
    float c[BM];     // w_i / (G Z_i)
    float mass[BM];  // V_i / Z_i
    int max_pos;
    int is_last;
    float tile_mass;
};

// Element offset of 16-byte chunk `ch` of row `row` in a [rows][D] bf16 tile
// whose chunks are XOR-swizzled by the low 3 row bits (conflict-free ldmatrix).
template <int D>
__device__ __forceinline__ int swz(int row, int ch) {
    return row * D + ((ch ^ (row & 7)) << 3);
}

// acc[nb][.] = 16 rows (this warp) x 64 keys of q k^T, fp32.
template <int D>
__device__ __forceinline__ void qk_tile(float (&acc)[8][4], const uint32_t (&qf)[D / 16][4],
                                        const uint16_t* sk, int lane) {
#pragma unroll
    for (int nb = 0; nb < 8; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[nb][e] = 0.f;
#pragma unroll
    for (int kc = 0; kc < D / 16; ++kc) {
#pragma unroll
        for (int pr = 0; pr < 4; ++pr) {
            const int row = pr * 16 + (lane & 7) + ((lane >> 4) << 3);
            const int ch = kc * 2 + ((lane >> 3) & 1);
            uint32_t b0, b1, b2, b3;
            ldsm_x4(smem_u32(sk + swz<D>(row, ch)), b0, b1, b2, b3);
            mma_bf16_16816(acc[2 * pr], qf[kc], b0, b1);
            mma_bf16_16816(acc[2 * pr + 1], qf[kc], b2, b3);
        }
    }
}

template <int D>
__global__ void __launch_bounds__(NTHREAD, 2)
score_stream_kernel(Problem p, const uint16_t* __restrict__ q, const uint16_t* __restrict__ k,
                    const uint8_t* __restrict__ modality, const int32_t* __restrict__ text_pos,
                    const float* __restrict__ w, float* __restrict__ scores,
                    float* __restrict__ tvb_stat, float* __restrict__ score_part,
                    float* __restrict__ stat_part, float* __restrict__ stat_head,
                    uint32_t* __restrict__ tickets, uint32_t* __restrict__ status) {
    extern __shared__ __align__(128) unsigned char smem_raw[];
    StreamSmem<D>& s = *reinterpret_cast<StreamSmem<D>*>(smem_raw);
    constexpr int CH = D / 8;  // 16-byte chunks per row

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int lh = blockIdx.y, l = lh / p.H_kv, g = lh % p.H_kv, t = blockIdx.x;
    const int row0 = t * BM;
    const bool first_cta = blockIdx.x == 0 && blockIdx.y == 0;

    // ---- query rows of this tile: positions and weights
    if (first_cta) {
        for (int i = tid; i < p.n_win; i += NTHREAD) {
            const int pi = text_pos[i];
            if (pi < 0 || pi >= p.N || (i > 0 && text_pos[i - 1] >= pi))
                raise_status(status, TGVKV_STATUS_TEXT_POS);
        }
    }
    if (tid == 0) s.max_pos = -1;
    if (tid < BM) {
        const int r = row0 + tid;
        int pos = -1;
        float wr = 0.f;
        if (r < p.R) {
            const int i = r % p.n_win;
            pos = text_pos[i];
            if (pos < 0 || pos >= p.N) pos = -1;  // reported above; the row is dropped
            wr = w[(long long)l * p.w_stride + i];
        }
        s.pos[tid] = pos;
        s.wrow[tid] = wr;
    }
    // ---- vision keys per key tile, then an exclusive scan -> vis_before
    const int n_tiles_all = (p.N + BN - 1) / BN;
    for (int kt = warp; kt < n_tiles_all; kt += NWARP) {
        const int j = kt * BN + lane;
        const bool v0 = j < p.N && modality[j] != 0;
        const bool v1 = j + 32 < p.N && modality[j + 32] != 0;
        const int cnt = __popc(__ballot_sync(~0u, v0)) + __popc(__ballot_sync(~0u, v1));
        if (lane == 0) s.vis_before[kt] = cnt;
    }
    __syncthreads();
    if (tid < BM) atomicMax(&s.max_pos, s.pos[tid]);
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
        if (lane == 0) s.vis_before[n_tiles_all] = total;
        if (lane == 0 && first_cta && total != p.N_v) raise_status(status, TGVKV_STATUS_VISION_COUNT);
    }
    __syncthreads();

    const int n_end = s.max_pos + 1;                 // keys 0..max_pos are visible to some row
    const int n_tiles = (n_end + BN - 1) / BN;
    const float sl2 = p.scale_log2;

    // ---- Q tile -> shared memory (rows past R are zero)
    const uint16_t* qbase = q + (size_t)(l * p.H_q + g * p.G) * p.n_win * D;
    for (int c = tid; c < BM * CH; c += NTHREAD) {
        const int row = c / CH, ch = c % CH;
        const int r = row0 + row;
        if (r < p.R)
            cp_async_16(smem_u32(&s.q[swz<D>(row, ch)]), qbase + (size_t)r * D + ch * 8);
        else
            *reinterpret_cast<uint4*>(&s.q[swz<D>(row, ch)]) = make_uint4(0, 0, 0, 0);
    }
    cp_async_commit();

    const uint16_t* kbase = k + (size_t)lh * p.N * D;
    auto load_k = [&](int kt, int buf) {
        const int j0 = kt * BN;
        for (int c = tid; c < BN * CH; c += NTHREAD) {
            const int row = c / CH, ch = c % CH;
            const int j = min(j0 + row, p.N - 1);   // rows past N are masked anyway
            cp_async_16(smem_u32(&s.k[buf][swz<D>(row, ch)]), kbase + (size_t)j * D + ch * 8);
        }
        if (warp == 0) {
            const int j = j0 + lane;
            const bool v0 = j < p.N && modality[j] != 0;
            const bool v1 = j + 32 < p.N && modality[j + 32] != 0;
            const unsigned b0 = __ballot_sync(~0u, v0), b1 = __ballot_sync(~0u, v1);
            const unsigned lt = (1u << lane) - 1u;
            const int base = s.vis_before[kt];
            s.vr[buf][lane] = v0 ? base + __popc(b0 & lt) : -1;
            s.vr[buf][lane + 32] = v1 ? base + __popc(b0) + __popc(b1 & lt) : -1;
        }
    };

    if (n_tiles > 0) load_k(0, 0);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();

    // ---- this warp's rows and Q fragments
    const int tq = lane & 3;
    const int rA = warp * 16 + (lane >> 2), rB = rA + 8;
    const int posA = s.pos[rA], posB = s.pos[rB];
    int wmax = max(posA, posB);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) wmax = max(wmax, __shfl_xor_sync(~0u, wmax, o));

    uint32_t qf[D / 16][4];
#pragma unroll
    for (int kc = 0; kc < D / 16; ++kc) {
        const int row = warp * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int ch = kc * 2 + (lane >> 4);
        ldsm_x4(smem_u32(&s.q[swz<D>(row, ch)]), qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3]);
    }

    // ---- pass A: online row statistics over every visible key
    float mA = -INFINITY, mB = -INFINITY, zA = 0.f, zB = 0.f, vA = 0.f, vB = 0.f;
    for (int kt = 0; kt < n_tiles; ++kt) {
        if (kt + 1 < n_tiles) load_k(kt + 1, (kt + 1) & 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const int buf = kt & 1, j0 = kt * BN;
        if (j0 <= wmax) {
            float acc[8][4];
            qk_tile<D>(acc, qf, s.k[buf], lane);
            float tA = -INFINITY, tB = -INFINITY;
#pragma unroll
            for (int nb = 0; nb < 8; ++nb)
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) {
                    const int j = j0 + nb * 8 + 2 * tq + cc;
                    const float xa = (j <= posA) ? acc[nb][cc] * sl2 : -INFINITY;
                    const float xb = (j <= posB) ? acc[nb][2 + cc] * sl2 : -INFINITY;
                    acc[nb][cc] = xa;
                    acc[nb][2 + cc] = xb;
                    tA = fmaxf(tA, xa);
                    tB = fmaxf(tB, xb);
                }
            tA = fmaxf(tA, __shfl_xor_sync(~0u, tA, 1));
            tA = fmaxf(tA, __shfl_xor_sync(~0u, tA, 2));
            tB = fmaxf(tB, __shfl_xor_sync(~0u, tB, 1));
            tB = fmaxf(tB, __shfl_xor_sync(~0u, tB, 2));
            const float nA = fmaxf(mA, tA), nB = fmaxf(mB, tB);
            const float uA = (nA == -INFINITY) ? 0.f : nA;
            const float uB = (nB == -INFINITY) ? 0.f : nB;
            const float aA = fast_exp2(mA - uA), aB = fast_exp2(mB - uB);
            zA *= aA; vA *= aA; zB *= aB; vB *= aB;
#pragma unroll
            for (int nb = 0; nb < 8; ++nb)
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) {
                    const bool vis = s.vr[buf][nb * 8 + 2 * tq + cc] >= 0;
                    const float ea = fast_exp2(acc[nb][cc] - uA);
                    const float eb = fast_exp2(acc[nb][2 + cc] - uB);
                    zA += ea; zB += eb;
                    if (vis) { vA += ea; vB += eb; }
                }
            mA = nA;
            mB = nB;
        }
        __syncthreads();
    }

    // ---- row statistics -> per-row factors
    zA += __shfl_xor_sync(~0u, zA, 1); zA += __shfl_xor_sync(~0u, zA, 2);
    zB += __shfl_xor_sync(~0u, zB, 1); zB += __shfl_xor_sync(~0u, zB, 2);
    vA += __shfl_xor_sync(~0u, vA, 1); vA += __shfl_xor_sync(~0u, vA, 2);
    vB += __shfl_xor_sync(~0u, vB, 1); vB += __shfl_xor_sync(~0u, vB, 2);
    const float inv_g = 1.f / (float)p.G;
    const bool okA = posA >= 0 && zA > 0.f, okB = posB >= 0 && zB > 0.f;
    const float cA = okA ? s.wrow[rA] * inv_g / zA : 0.f;
    const float cB = okB ? s.wrow[rB] * inv_g / zB : 0.f;
    const float uA = (mA == -INFINITY) ? 0.f : mA;
    const float uB = (mB == -INFINITY) ? 0.f : mB;
    if (tq == 0) {
        s.mass[rA] = okA ? vA / zA : 0.f;
        s.mass[rB] = okB ? vB / zB : 0.f;
    }
    __syncthreads();
    if (tid == 0) {
        float acc = 0.f;
        for (int r = 0; r < BM; ++r) acc += s.mass[r];
        s.tile_mass = acc;
    }

    // ---- pass B: text-weighted column sums over the vision keys
    float* out = (p.T == 1) ? scores + (size_t)lh * p.N_v
                            : score_part + ((size_t)lh * p.T + t) * p.N_v;
    auto next_vis = [&](int kt) {
        while (kt < n_tiles && s.vis_before[kt + 1] == s.vis_before[kt]) ++kt;
        return kt;
    };
    int kt = next_vis(0);
    int buf = 0;
    if (kt < n_tiles) load_k(kt, 0);
    cp_async_commit();
    while (kt < n_tiles) {
        const int kn = next_vis(kt + 1);
        if (kn < n_tiles) load_k(kn, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const int j0 = kt * BN;
        float u[16];
        if (j0 <= wmax) {
            float acc[8][4];
            qk_tile<D>(acc, qf, s.k[buf], lane);
#pragma unroll
            for (int nb = 0; nb < 8; ++nb)
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) {
                    const int col = nb * 8 + 2 * tq + cc;
                    const int j = j0 + col;
                    const bool vis = s.vr[buf][col] >= 0;
                    const float pa = (vis && j <= posA) ? cA * fast_exp2(acc[nb][cc] * sl2 - uA) : 0.f;
                    const float pb = (vis && j <= posB) ? cB * fast_exp2(acc[nb][2 + cc] * sl2 - uB) : 0.f;
                    u[nb * 2 + cc] = pa + pb;
                }
            // sum over the 8 lanes that share tq (16 rows): transpose-reduce,
            // leaving two column sums per lane
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const bool hi = lane & 16;
                const float send = hi ? u[i] : u[i + 8];
                const float keep = hi ? u[i + 8] : u[i];
                u[i] = keep + __shfl_xor_sync(~0u, send, 16);
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const bool hi = lane & 8;
                const float send = hi ? u[i] : u[i + 4];
                const float keep = hi ? u[i + 4] : u[i];
                u[i] = keep + __shfl_xor_sync(~0u, send, 8);
            }
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const bool hi = lane & 4;
                const float send = hi ? u[i] : u[i + 2];
                const float keep = hi ? u[i + 2] : u[i];
                u[i] = keep + __shfl_xor_sync(~0u, send, 4);
            }
        } else {
            u[0] = 0.f;
            u[1] = 0.f;
        }
        {
            const int nb = ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1);
            s.colsum[warp][nb * 8 + 2 * tq] = u[0];
            s.colsum[warp][nb * 8 + 2 * tq + 1] = u[1];
        }
        __syncthreads();
        if (tid < BN) {
            const int vr = s.vr[buf][tid];
            if (vr >= 0 && vr < p.N_v) {
                float a = 0.f;
#pragma unroll
                for (int ww = 0; ww < NWARP; ++ww) a += s.colsum[ww][tid];
                out[vr] = a;
            }
        }
        __syncthreads();
        kt = kn;
        buf ^= 1;
    }
    // vision keys after every query row of this tile: zero attention
    for (int v = s.vis_before[n_tiles] + tid; v < p.N_v; v += NTHREAD) out[v] = 0.f;

    // ---- reductions over row tiles (per head) and heads (per layer)
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
        for (int v = tid; v < p.N_v; v += NTHREAD) {
            float a = 0.f;
            for (int tt = 0; tt < p.T; ++tt) a += __ldcg(&score_part[((size_t)lh * p.T + tt) * p.N_v + v]);
            scores[(size_t)lh * p.N_v + v] = a;
        }
        if (tid == 0) {
            float m = 0.f;
            for (int tt = 0; tt < p.T; ++tt) m += __ldcg(&stat_part[(size_t)lh * p.T + tt]);
            stat_head[lh] = m;
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

template <int D>
cudaError_t launch_stream(const Problem& p, const uint16_t* q, const uint16_t* k,
                          const uint8_t* modality, const int32_t* text_pos, const float* w,
                          float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                          cudaStream_t stream) {
    const size_t smem = sizeof(StreamSmem<D>);
    cudaError_t e = cudaFuncSetAttribute(score_stream_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid(p.T, p.L * p.H_kv);
    score_stream_kernel<D><<<grid, NTHREAD, smem, stream>>>(
        p, q, k, modality, text_pos, w, scores, tvb_stat,
        reinterpret_cast<float*>(ws + lay.score_part), reinterpret_cast<float*>(ws + lay.stat_part),
        reinterpret_cast<float*>(ws + lay.stat_head), reinterpret_cast<uint32_t*>(ws + lay.tickets),
        reinterpret_cast<uint32_t*>(ws + lay.status));
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score(const Problem& p, const uint16_t* q, const uint16_t* k,
                         const uint8_t* modality, const int32_t* text_pos, const float* w,
                         float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                         cudaStream_t stream) {
    cudaError_t e = cudaMemsetAsync(ws + lay.tickets, 0,
                                    sizeof(uint32_t) * (size_t)(p.L * p.H_kv + p.L), stream);
    if (e != cudaSuccess) return e;
    if (p.R == 0) {  // no query rows: no attention mass anywhere
        if (p.N_v > 0) {
            e = cudaMemsetAsync(scores, 0, sizeof(float) * (size_t)p.L * p.H_kv * p.N_v, stream);
            if (e != cudaSuccess) return e;
        }
        return cudaMemsetAsync(tvb_stat, 0, sizeof(float) * (size_t)p.L, stream);
    }
    return launch_score_tc(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
}

cudaError_t launch_score_stream(const Problem& p, const uint16_t* q, const uint16_t* k,
                                const uint8_t* modality, const int32_t* text_pos, const float* w,
                                float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                                cudaStream_t stream) {
    if (p.d == 64)
        return launch_stream<64>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
    return launch_stream<128>(p, q, k, modality, text_pos, w, scores, tvb_stat, ws, lay, stream);
}

}  // namespace tgvkv
