// TPR retention (Eq. 10).  The hot path (vision basis, no sinks) is the case
// b_l > N_t with the vision budget b_l: one CTA per
// (layer, KV head) keeps every text position and the b_l vision positions of
// highest score, ties to the lower position, in ascending position order --
// and, in the fused form used by tgvkv_evict, gathers the retained K and V
// rows straight away.  The layer budgets come in from global memory (on the
// evict path the score kernel derives them).
//
// In the fused form the rows of the text runs before the first and after the
// last vision key ("edge" rows) have slots that the budget alone fixes (the
// first rows and the last rows of the set), so extra CTAs copy them while the
// selecting CTAs select; a selecting CTA gathers the interior rows only.
//
// Selection: the scores become order-preserving 32-bit keys in shared memory;
// an MSB-first radix select (four 8-bit digits) finds the key T of the b_l-th
// largest score and how many keys equal to T are still needed (k_eq).  A
// vision key is kept iff key > T, or key == T and it is among the first k_eq
// such keys in position order.  When every key equal to T is kept (the last
// round's bin holds exactly k_eq keys, the usual case), keep = key >= T and
// each warp walks a contiguous range of positions with ballots, two block
// prefix sums giving the ranges their vision rank and output slot bases;
// with ties to break, each thread owns a range and three block prefix sums
// (vision keys, keys equal to T, kept positions) give the slots.
#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kThreads = 256;
constexpr size_t kFusedSmemLimit = 200 * 1024; // keys + retained rows held for the gather

// Exclusive prefix sum of x over the block; *total gets the block sum.
__device__ __forceinline__ int block_exclusive_scan(int x, int* buf, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(~0u, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) buf[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int v = (lane < kThreads / 32) ? buf[lane] : 0;
        int iv = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(~0u, iv, o);
            if (lane >= o) iv += y;
        }
        buf[lane] = iv - v;
        if (lane == 31) buf[32] = iv;
    }
    __syncthreads();
    const int res = buf[warp] + incl - x;
    *total = buf[32];
    __syncthreads();
    return res;
}

// First vision position (N if none) and one past the last (0 if none) of the
// modality bytes in shared memory, reduced over the block.
__device__ __forceinline__ void vision_span_block(const uint8_t* modality, int N, int* lo, int* hi,
                                                  int* red) {
    int a = N, z = 0;
    for (int j = threadIdx.x; j < N; j += blockDim.x)
        if (modality[j]) {
            a = min(a, j);
            z = max(z, j + 1);
        }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        a = min(a, __shfl_xor_sync(~0u, a, o));
        z = max(z, __shfl_xor_sync(~0u, z, o));
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    if (lane == 0) {
        red[warp] = a;
        red[32 + warp] = z;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < nw; ++w) {
            red[0] = min(red[0], red[w]);
            red[32] = max(red[32], red[32 + w]);
        }
    }
    __syncthreads();
    *lo = red[0];
    *hi = red[32];
    __syncthreads();
}

// Copy `rows` consecutive K and V rows of head `head` starting at position
// `src0` to output rows starting at `dst0`, with the threads [t0, t0 + nt)
// (16-byte vectors, loads before stores).
template <int VPR>
__device__ __forceinline__ void copy_rows(const uint4* __restrict__ k, const uint4* __restrict__ v,
                                          uint4* __restrict__ k_out, uint4* __restrict__ v_out,
                                          size_t head, int src0, long long dst0, int rows, int t,
                                          int nt) {
    constexpr int UNROLL = 4;
    const int nvec = rows * VPR;
    for (int i0 = t; i0 < nvec; i0 += nt * UNROLL) {
        uint4 kr[UNROLL], vr[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int i = i0 + u * nt;
            if (i < nvec) {
                kr[u] = __ldg(k + (head + src0) * VPR + i);
                vr[u] = __ldg(v + (head + src0) * VPR + i);
            }
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int i = i0 + u * nt;
            if (i < nvec) {
                k_out[(size_t)dst0 * VPR + i] = kr[u];
                v_out[(size_t)dst0 * VPR + i] = vr[u];
            }
        }
    }
}

// Shared memory of one CTA: keys [N_v], retained rows [N] (gather form) and
// the modality bytes [N].
__host__ __device__ inline size_t select_smem(const Problem& p, bool compact) {
    return sizeof(uint32_t) * (size_t)p.N_v + (compact ? sizeof(int) * (size_t)p.N : 0) +
           (((size_t)p.N + 15) & ~size_t(15));
}

// COMPACT: also gather the retained rows.
// (Register bounds: five CTAs per SM in the fused form, eight in the select-only form.)
template <bool COMPACT, int VPR>
__global__ void __launch_bounds__(kThreads, COMPACT ? 5 : 8)
tpr_select_kernel(Problem p, const float* __restrict__ scores, const int32_t* __restrict__ budgets,
                  const uint8_t* __restrict__ modality_g, int64_t* __restrict__ offsets,
                  int32_t* __restrict__ idx, const uint4* __restrict__ k,
                  const uint4* __restrict__ v, uint4* __restrict__ k_out,
                  uint4* __restrict__ v_out, long long capacity, uint32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char dyn_raw[];
    uint32_t* keys = reinterpret_cast<uint32_t*>(dyn_raw);  // [N_v]
    int* rows = reinterpret_cast<int*>(keys + p.N_v);       // [N_t + b] (gather form)
    uint8_t* modality = reinterpret_cast<uint8_t*>(dyn_raw) + sizeof(uint32_t) * (size_t)p.N_v +
                        (COMPACT ? sizeof(int) * (size_t)p.N : 0);   // [N]
    __shared__ int hist[256];
    __shared__ int scan_buf[33];
    __shared__ uint32_t s_prefix;
    __shared__ int s_kk;
    __shared__ int s_ties;

    // a kernel after this one (the next eviction's score kernel) reads nothing
    // this one writes: it may be scheduled once every CTA of this grid has begun
    if (COMPACT) griddep_launch_dependents();
    // fused form: CTA 2h selects head h and gathers its interior rows, CTA
    // 2h + 1 copies its edge rows
    const int lg = COMPACT ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
    const bool edge_cta = COMPACT && (blockIdx.x & 1);
    const int l = lg / p.H_kv, g = lg % p.H_kv;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ int span_red[64];

    for (int j = tid; j < p.N; j += kThreads) modality[j] = __ldg(modality_g + j);
    __syncthreads();
    int vlo = 0, vhi = 0;   // edge rows: positions [0, vlo) and [vhi, N)
    if (COMPACT) vision_span_block(modality, p.N, &vlo, &vhi, span_red);
    if (vhi < vlo) vhi = vlo;   // no vision key: every row is a leading edge row
    // the scores and budgets come from the kernel before (as a programmatic
    // dependent of the score kernel, this CTA may have started while its last
    // CTA split the budgets): wait, then read them through L2
    griddep_wait();
    int b = __ldcg(budgets + l);
    if (b < 0 || b > p.N_v) {
        if (tid == 0) raise_status(status, TGVKV_STATUS_BUDGET);
        b = b < 0 ? 0 : p.N_v;
    }
    const int len = p.N_t + b;
    // CSR offset: the sets of the earlier layers, summed by the whole block
    // (their budgets load in parallel, not one after another)
    __shared__ long long off_part[kThreads / 32];
    {
        long long part = 0;
        for (int m = tid; m < l; m += kThreads) {
            int bm = __ldcg(budgets + m);
            bm = bm < 0 ? 0 : (bm > p.N_v ? p.N_v : bm);
            part += (long long)p.H_kv * (p.N_t + bm);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(~0u, part, o);
        if (lane == 0) off_part[warp] = part;
    }
    __syncthreads();
    // the set's first row, the same in every thread (recomputed where needed
    // rather than held in registers across the selection)
    auto set_offset = [&]() {
        long long o = (long long)g * len;
        for (int w = 0; w < kThreads / 32; ++w) o += off_part[w];
        return o;
    };
    // a set that would end past the caller's rows writes none of its rows or indices
    const bool fits = set_offset() + len <= capacity;
    if (edge_cta) {
        if (!fits) return;
        const long long off = set_offset();
        const size_t head = (size_t)lg * p.N;
        const int tail = p.N - vhi;
        if (vlo <= len) copy_rows<VPR>(k, v, k_out, v_out, head, 0, off, vlo, tid, kThreads);
        if (tail <= len - vlo)
            copy_rows<VPR>(k, v, k_out, v_out, head, vhi, off + len - tail, tail, tid, kThreads);
        return;
    }
    if (tid == 0) {
        const long long off = set_offset();
        offsets[lg] = off;
        if (lg == p.L * p.H_kv - 1) offsets[lg + 1] = off + len;
        if (!fits) raise_status(status, TGVKV_STATUS_INDEX);
    }
    if (!fits) return;
    const float* sc = scores + (size_t)lg * p.N_v;
    for (int i = tid; i < p.N_v; i += kThreads) keys[i] = float_order_key(__ldcg(sc + i));
    __syncthreads();

    // ---- radix select of the b-th largest key
    uint32_t prefix = 0;
    int kk = b;
    if (b > 0) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            hist[tid] = 0;   // kThreads == 256 bins
            __syncthreads();
            const uint32_t hi_mask = (shift == 24) ? 0u : (0xFFFFFFFFu << (shift + 8));
            for (int i = tid; i < p.N_v; i += kThreads) {
                const uint32_t key = keys[i];
                if ((key & hi_mask) == (prefix & hi_mask)) atomicAdd(&hist[(key >> shift) & 255], 1);
            }
            __syncthreads();
            if (warp == 0) {
                // lane 0 holds the 8 highest digits, lane 31 the 8 lowest
                int cnt[8];
                int sum = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    cnt[e] = hist[255 - 8 * lane - e];
                    sum += cnt[e];
                }
                int incl = sum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(~0u, incl, o);
                    if (lane >= o) incl += y;
                }
                const int above = incl - sum;
                if (above < kk && kk <= above + sum) {
                    int a = above;
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        if (kk <= a + cnt[e]) {
                            s_prefix = prefix | ((uint32_t)(255 - 8 * lane - e) << shift);
                            s_kk = kk - a;
                            s_ties = cnt[e];   // after the last round: the keys equal to T
                            break;
                        }
                        a += cnt[e];
                    }
                }
            }
            __syncthreads();
            prefix = s_prefix;
            kk = s_kk;
        }
    }
    const bool none = (b == 0);
    const uint32_t thr = prefix;
    const int k_eq = none ? 0 : kk;
    int tot;
    const long long off = set_offset();

    if (none || s_ties == k_eq) {
        // ---- every key equal to T is kept (no ties to break): a vision key
        // is kept iff key >= T.  Each warp owns a contiguous range of
        // positions and walks it 32 at a time with ballots; two block scans
        // give the ranges their vision rank and output slot bases.
        const uint32_t lt = (1u << lane) - 1u;
        constexpr int kWarps = kThreads / 32;
        const int wper = (((p.N + kWarps - 1) / kWarps) + 31) & ~31;
        const int w0 = min(p.N, warp * wper), w1 = min(p.N, w0 + wper);
        int nvw = 0;
        for (int c0 = w0; c0 < w1; c0 += 32) {
            const int j = c0 + lane;
            nvw += __popc(__ballot_sync(~0u, j < w1 && modality[j] != 0));
        }
        const int vbase = __shfl_sync(~0u, block_exclusive_scan(lane == 0 ? nvw : 0, scan_buf, &tot), 0);
        auto walk = [&](auto&& emit) {
            int vr = vbase, kr = 0;
            for (int c0 = w0; c0 < w1; c0 += 32) {
                const int j = c0 + lane;
                const bool in = j < w1;
                const bool isv = in && modality[j] != 0;
                const uint32_t vb = __ballot_sync(~0u, isv);
                const int myvr = vr + __popc(vb & lt);
                const bool keep = in && (!isv || (!none && myvr < p.N_v && keys[myvr] >= thr));
                const uint32_t kb = __ballot_sync(~0u, keep);
                if (keep) emit(j, kr + __popc(kb & lt));
                vr += __popc(vb);
                kr += __popc(kb);
            }
            return kr;
        };
        const int nkw = walk([](int, int) {});
        const int kbase = __shfl_sync(~0u, block_exclusive_scan(lane == 0 ? nkw : 0, scan_buf, &tot), 0);
        walk([&](int j, int rr) {
            const int r = kbase + rr;
            if (r < len) {
                idx[off + r] = j;
                if (COMPACT) rows[r] = j;
            }
        });
    } else {
        // ---- ties at T to break: ordered emission over per-thread position
        // ranges, the first k_eq keys equal to T (in position order) kept
        const int per = (p.N + kThreads - 1) / kThreads;
        const int j0 = min(p.N, tid * per), j1 = min(p.N, j0 + per);
        int nv = 0;
        for (int j = j0; j < j1; ++j) nv += modality[j] != 0;
        const int vbase = block_exclusive_scan(nv, scan_buf, &tot);
        int neq = 0;
        if (!none) {
            int vr = vbase;
            for (int j = j0; j < j1; ++j)
                if (modality[j] != 0) {
                    neq += (vr < p.N_v && keys[vr] == thr);
                    ++vr;
                }
        }
        const int ebase = block_exclusive_scan(neq, scan_buf, &tot);
        // kept(j): text, or a vision key above T, or one of the first k_eq equal to T
        auto scan_kept = [&](auto&& emit) {
            int vr = vbase, er = ebase;
            for (int j = j0; j < j1; ++j) {
                bool keep = true;
                if (modality[j] != 0) {
                    keep = false;
                    if (vr < p.N_v && !none) {
                        const uint32_t key = keys[vr];
                        if (key > thr) {
                            keep = true;
                        } else if (key == thr) {
                            keep = er < k_eq;
                            ++er;
                        }
                    }
                    ++vr;
                }
                if (keep) emit(j);
            }
        };
        int nkeep = 0;
        scan_kept([&](int) { ++nkeep; });
        const int kbase = block_exclusive_scan(nkeep, scan_buf, &tot);
        {
            int r = kbase;
            scan_kept([&](int j) {
                if (r < len) {
                    idx[off + r] = j;
                    if (COMPACT) rows[r] = j;
                }
                ++r;
            });
        }
    }
    if (tid == 0 && tot != len) raise_status(status, TGVKV_STATUS_COUNT);
    if (!COMPACT) return;

    // ---- gather the interior retained K and V rows (fused form): the set's
    // first vlo rows and last N - vhi rows are the edge CTA's
    __syncthreads();
    constexpr int RPI = 32 / VPR;     // rows per warp per step
    constexpr int UNROLL = 4;
    const bool edges_ok = vlo <= len && p.N - vhi <= len - vlo;
    const int n = min(len, tot) - (edges_ok ? p.N - vhi : 0);
    const int rfirst = edges_ok ? vlo : 0;
    const int sub = lane / VPR, vec = lane % VPR;
    const size_t head = (size_t)lg * p.N;
    for (int r0 = rfirst + warp * RPI * UNROLL; r0 < n; r0 += (kThreads / 32) * RPI * UNROLL) {
        uint4 kr[UNROLL], vr[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int r = r0 + u * RPI + sub;
            if (r < n) {
                const size_t src = (head + rows[r]) * VPR + vec;
                kr[u] = __ldg(k + src);
                vr[u] = __ldg(v + src);
            }
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int r = r0 + u * RPI + sub;
            if (r < n) {
                const size_t dst = (size_t)(off + r) * VPR + vec;
                k_out[dst] = kr[u];
                v_out[dst] = vr[u];
            }
        }
    }
}

// ---- warp per (layer, KV head): select, emit and gather with warp-level
// synchronisation only.  For shapes with many small heads: the warps of an SM
// work on different heads and drift apart, so one warp's selection overlaps
// other warps' gathers.  Shared memory per warp: keys [N_v], a 256-bin
// histogram and the retained rows [N]; the modality bytes are shared by the CTA.
__host__ __device__ inline size_t warp_select_words(const Problem& p) {
    return (size_t)p.N_v + 256 + (size_t)p.N;
}

template <int VPR>
__global__ void __launch_bounds__(256)
tpr_select_warp_kernel(Problem p, const float* __restrict__ scores,
                       const int32_t* __restrict__ budgets, const uint8_t* __restrict__ modality_g,
                       int64_t* __restrict__ offsets, int32_t* __restrict__ idx,
                       const uint4* __restrict__ k, const uint4* __restrict__ v,
                       uint4* __restrict__ k_out, uint4* __restrict__ v_out,
                       long long capacity, uint32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char dyn_raw[];
    const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nw = blockDim.x >> 5;
    // a kernel after this one (the next eviction's score kernel) reads nothing
    // this one writes: it may be scheduled once every CTA of this grid has begun
    griddep_launch_dependents();
    const size_t mod_bytes = ((size_t)p.N + 15) & ~size_t(15);
    uint8_t* modality = dyn_raw;
    uint32_t* keys = reinterpret_cast<uint32_t*>(dyn_raw + mod_bytes) + (size_t)wid * warp_select_words(p);
    int* hist = reinterpret_cast<int*>(keys + p.N_v);
    int* rows = hist + 256;
    for (int j = threadIdx.x; j < p.N; j += blockDim.x) modality[j] = __ldg(modality_g + j);
    __syncthreads();
    // CTA 2c selects and gathers the interior rows of heads c*nw.., CTA 2c + 1
    // copies their edge rows (positions [0, vlo) and [vhi, N))
    __shared__ int span_red[64];
    int vlo, vhi;
    vision_span_block(modality, p.N, &vlo, &vhi, span_red);
    if (vhi < vlo) vhi = vlo;
    // the scores and budgets come from the kernel before: wait, then read them through L2
    griddep_wait();
    const bool edge_cta = blockIdx.x & 1;
    const int lg = (int)(blockIdx.x >> 1) * nw + wid;
    if (lg >= p.L * p.H_kv) return;
    const int l = lg / p.H_kv, g = lg % p.H_kv;
    const uint32_t lt = (1u << lane) - 1u;

    int b = __ldcg(budgets + l);
    if (b < 0 || b > p.N_v) {
        if (lane == 0) raise_status(status, TGVKV_STATUS_BUDGET);
        b = b < 0 ? 0 : p.N_v;
    }
    const int len = p.N_t + b;
    // CSR offset: rows of every (layer, head) before this one
    long long off = 0;
    for (int m = lane; m < l; m += 32) {
        int bm = __ldcg(budgets + m);
        bm = bm < 0 ? 0 : (bm > p.N_v ? p.N_v : bm);
        off += (long long)p.H_kv * (p.N_t + bm);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) off += __shfl_xor_sync(~0u, off, o);
    off += (long long)g * len;
    const int tail = p.N - vhi;
    const bool edges_ok = vlo <= len && tail <= len - vlo;
    // a set that would end past the caller's rows writes none of its rows or indices
    const bool fits = off + len <= capacity;
    if (edge_cta) {
        if (edges_ok && fits) {
            const size_t head = (size_t)lg * p.N;
            copy_rows<VPR>(k, v, k_out, v_out, head, 0, off, vlo, lane, 32);
            copy_rows<VPR>(k, v, k_out, v_out, head, vhi, off + len - tail, tail, lane, 32);
        }
        return;
    }
    if (lane == 0) {
        offsets[lg] = off;
        if (lg == p.L * p.H_kv - 1) offsets[lg + 1] = off + len;
        if (!fits) raise_status(status, TGVKV_STATUS_INDEX);
    }
    if (!fits) return;
    const float* sc = scores + (size_t)lg * p.N_v;
    for (int i = lane; i < p.N_v; i += 32) keys[i] = float_order_key(__ldcg(sc + i));
    __syncwarp();

    // ---- radix select of the b-th largest key, 8 bits per round
    uint32_t prefix = 0;
    int kk = b;
    if (b > 0) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            for (int i = lane; i < 256; i += 32) hist[i] = 0;
            __syncwarp();
            const uint32_t hi_mask = (shift == 24) ? 0u : (0xFFFFFFFFu << (shift + 8));
            for (int i = lane; i < p.N_v; i += 32) {
                const uint32_t key = keys[i];
                if ((key & hi_mask) == (prefix & hi_mask)) atomicAdd(&hist[(key >> shift) & 255], 1);
            }
            __syncwarp();
            // lane t holds digits 255-8t .. 248-8t (highest first)
            int cnt[8];
            int sum = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                cnt[e] = hist[255 - 8 * lane - e];
                sum += cnt[e];
            }
            int incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(~0u, incl, o);
                if (lane >= o) incl += y;
            }
            const int above = incl - sum;
            const bool here = above < kk && kk <= above + sum;
            uint32_t digit = 0;
            int rest = 0;
            if (here) {
                int a = above;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (kk <= a + cnt[e]) {
                        digit = (uint32_t)(255 - 8 * lane - e);
                        rest = kk - a;
                        break;
                    }
                    a += cnt[e];
                }
            }
            const int src = __ffs(__ballot_sync(~0u, here)) - 1;   // exactly one lane
            digit = __shfl_sync(~0u, digit, src < 0 ? 0 : src);
            rest = __shfl_sync(~0u, rest, src < 0 ? 0 : src);
            prefix |= digit << shift;
            kk = rest;
            __syncwarp();
        }
    }
    const bool none = (b == 0);
    const uint32_t thr = prefix;
    const int k_eq = none ? 0 : kk;

    // ---- emission in position order, 32 positions per round
    int vr_base = 0, eq_base = 0, out_base = 0;
    for (int c0 = 0; c0 < p.N; c0 += 32) {
        const int j = c0 + lane;
        const bool in = j < p.N;
        const bool isv = in && modality[j] != 0;
        const uint32_t vb = __ballot_sync(~0u, isv);
        const int vr = vr_base + __popc(vb & lt);
        bool keep = in && !isv, eq = false;
        if (isv && !none && vr < p.N_v) {
            const uint32_t key = keys[vr];
            if (key > thr) keep = true;
            else if (key == thr) eq = true;
        }
        const uint32_t eb = __ballot_sync(~0u, eq);
        if (eq && eq_base + __popc(eb & lt) < k_eq) keep = true;
        const uint32_t kb = __ballot_sync(~0u, keep);
        const int r = out_base + __popc(kb & lt);
        if (keep && r < len) {
            idx[off + r] = j;
            rows[r] = j;
        }
        vr_base += __popc(vb);
        eq_base += __popc(eb);
        out_base += __popc(kb);
    }
    if (lane == 0 && out_base != len) raise_status(status, TGVKV_STATUS_COUNT);
    __syncwarp();

    // ---- gather the interior retained K and V rows (the edge CTA copies the rest)
    constexpr int RPI = 32 / VPR;   // rows per warp instruction
    constexpr int UNROLL = 8;
    const int n = min(len, out_base) - (edges_ok ? tail : 0);
    const int rfirst = edges_ok ? vlo : 0;
    const int sub = lane / VPR, vec = lane % VPR;
    const size_t head = (size_t)lg * p.N;
    for (int r0 = rfirst; r0 < n; r0 += RPI * UNROLL) {
        uint4 kr[UNROLL], vr[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int r = r0 + u * RPI + sub;
            if (r < n) {
                const size_t src = (head + rows[r]) * VPR + vec;
                kr[u] = __ldg(k + src);
                vr[u] = __ldg(v + src);
            }
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int r = r0 + u * RPI + sub;
            if (r < n) {
                const size_t dst = (size_t)(off + r) * VPR + vec;
                k_out[dst] = kr[u];
                v_out[dst] = vr[u];
            }
        }
    }
}

// ---- the general form: both cases of Eq. 10 and sink tokens (any basis).
// Per layer the case is chosen by b_l: under the all-token basis b_l > N_t
// ranks the vision keys by the Eq. 8 score on top of every text key, and
// b_l <= N_t ranks the text keys by the Eq. 9 score with no vision key;
// under the vision basis the first case holds with b_l vision slots.  Sinks
// are always kept; a sink of the ranked modality takes one slot (its key is
// set to 0, below every score's key, so the radix select never picks it).
struct TprCase {
    bool vision;   // the ranked candidates are the vision keys
    int slots;     // candidates chosen by rank (sinks excluded)
    int len;       // retained rows of each head of the layer
};

__host__ __device__ inline TprCase tpr_case(const Problem& p, int b, int sink_v, int sink_t) {
    TprCase c;
    const bool all = p.basis == TGVKV_BASIS_ALL;
    c.vision = !all || b > p.N_t;
    const int n_cand = c.vision ? p.N_v : p.N_t;
    const int sink_c = c.vision ? sink_v : sink_t;
    int slots = (all && c.vision) ? b - p.N_t : b;
    slots -= sink_c;
    slots = slots < 0 ? 0 : (slots > n_cand - sink_c ? n_cand - sink_c : slots);
    c.slots = slots;
    c.len = (c.vision ? p.N_t + sink_v : sink_v + sink_t) + slots;
    return c;
}

__host__ __device__ inline int budget_cap_of(const Problem& p) {
    return p.basis == TGVKV_BASIS_ALL ? p.N : p.N_v;
}

__host__ __device__ inline size_t select_general_smem(const Problem& p, bool compact) {
    const size_t keyset = (size_t)(p.N_v > p.N_t ? p.N_v : p.N_t);
    return sizeof(uint32_t) * keyset + (compact ? sizeof(int) * (size_t)p.N : 0) +
           (((size_t)p.N + 15) & ~size_t(15));
}

template <bool COMPACT, int VPR>
__global__ void __launch_bounds__(kThreads)
tpr_select_general_kernel(Problem p, const float* __restrict__ scores,
                          const float* __restrict__ text_scores,
                          const int32_t* __restrict__ budgets, const uint8_t* __restrict__ modality_g,
                          int64_t* __restrict__ offsets, int32_t* __restrict__ idx,
                          const uint4* __restrict__ k, const uint4* __restrict__ v,
                          uint4* __restrict__ k_out, uint4* __restrict__ v_out,
                          long long capacity, uint32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char dyn_raw[];
    const size_t keyset = (size_t)(p.N_v > p.N_t ? p.N_v : p.N_t);
    uint32_t* keys = reinterpret_cast<uint32_t*>(dyn_raw);          // [candidates]
    int* rows = reinterpret_cast<int*>(keys + keyset);             // [len] (gather form)
    uint8_t* modality = reinterpret_cast<uint8_t*>(dyn_raw) + sizeof(uint32_t) * keyset +
                        (COMPACT ? sizeof(int) * (size_t)p.N : 0);   // [N]
    __shared__ int hist[256];
    __shared__ int scan_buf[33];
    __shared__ uint32_t s_prefix;
    __shared__ int s_kk, s_sink_v, s_sink_t;
    __shared__ long long s_off;

    const int lg = blockIdx.x, l = lg / p.H_kv, g = lg % p.H_kv;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        s_sink_v = 0;
        s_sink_t = 0;
    }
    __syncthreads();
    int sv = 0, st = 0;
    for (int j = tid; j < p.N; j += kThreads) {
        const uint8_t m = __ldg(modality_g + j);
        modality[j] = m;
        if (is_sink(p, j)) (m != 0 ? sv : st) += 1;
    }
    if (sv) atomicAdd(&s_sink_v, sv);
    if (st) atomicAdd(&s_sink_t, st);
    __syncthreads();
    const int sink_v = s_sink_v, sink_t = s_sink_t;
    const int cap = budget_cap_of(p);
    int b = budgets[p.head_budgets ? lg : l];
    if (b < 0 || b > cap) {
        if (tid == 0) raise_status(status, TGVKV_STATUS_BUDGET);
        b = b < 0 ? 0 : cap;
    }
    const TprCase c = tpr_case(p, b, sink_v, sink_t);
    const int len = c.len;
    if (p.head_budgets) {
        // CSR offset: the set sizes of every earlier head, summed by the block
        long long part = 0;
        for (int m = tid; m < lg; m += kThreads) {
            int bm = budgets[m];
            bm = bm < 0 ? 0 : (bm > cap ? cap : bm);
            part += tpr_case(p, bm, sink_v, sink_t).len;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(~0u, part, o);
        __shared__ long long warp_part[kThreads / 32];
        if (lane == 0) warp_part[warp] = part;
        __syncthreads();
        if (tid == 0) {
            long long off = 0;
            for (int w = 0; w < kThreads / 32; ++w) off += warp_part[w];
            s_off = off;
            offsets[lg] = off;
            if (lg == p.L * p.H_kv - 1) offsets[lg + 1] = off + len;
        }
    } else {
        // the sets of the earlier layers, summed by the whole block
        long long part = 0;
        for (int m = tid; m < l; m += kThreads) {
            int bm = budgets[m];
            bm = bm < 0 ? 0 : (bm > cap ? cap : bm);
            part += (long long)p.H_kv * tpr_case(p, bm, sink_v, sink_t).len;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(~0u, part, o);
        __shared__ long long layer_part[kThreads / 32];
        if (lane == 0) layer_part[warp] = part;
        __syncthreads();
        if (tid == 0) {
            long long off = (long long)g * len;
            for (int w = 0; w < kThreads / 32; ++w) off += layer_part[w];
            s_off = off;
            offsets[lg] = off;
            if (lg == p.L * p.H_kv - 1) offsets[lg + 1] = off + len;
        }
    }
    const int n_cand = c.vision ? p.N_v : p.N_t;
    const uint8_t cand_mod = c.vision ? 1 : 0;
    const float* sc = c.vision ? scores + (size_t)lg * p.N_v : text_scores + (size_t)lg * p.N_t;
    for (int i = tid; i < n_cand; i += kThreads) keys[i] = float_order_key(__ldg(sc + i));
    __syncthreads();
    // a set that would end past the caller's rows writes none of its rows or indices
    if (s_off + len > capacity) {
        if (tid == 0) raise_status(status, TGVKV_STATUS_INDEX);
        return;
    }

    // ---- candidate ranks of each thread's contiguous position range; sinks get key 0
    const int per = (p.N + kThreads - 1) / kThreads;
    const int j0 = min(p.N, tid * per), j1 = min(p.N, j0 + per);
    int nc = 0;
    for (int j = j0; j < j1; ++j) nc += (modality[j] != 0) == (cand_mod != 0);
    int tot;
    const int cbase = block_exclusive_scan(nc, scan_buf, &tot);
    {
        int cr = cbase;
        for (int j = j0; j < j1; ++j)
            if ((modality[j] != 0) == (cand_mod != 0)) {
                if (is_sink(p, j) && cr < n_cand) keys[cr] = 0u;
                ++cr;
            }
    }
    __syncthreads();

    // ---- radix select of the slots-th largest key
    uint32_t prefix = 0;
    int kk = c.slots;
    if (c.slots > 0) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            hist[tid] = 0;   // kThreads == 256 bins
            __syncthreads();
            const uint32_t hi_mask = (shift == 24) ? 0u : (0xFFFFFFFFu << (shift + 8));
            for (int i = tid; i < n_cand; i += kThreads) {
                const uint32_t key = keys[i];
                if ((key & hi_mask) == (prefix & hi_mask)) atomicAdd(&hist[(key >> shift) & 255], 1);
            }
            __syncthreads();
            if (warp == 0) {
                int cnt[8];
                int sum = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    cnt[e] = hist[255 - 8 * lane - e];
                    sum += cnt[e];
                }
                int incl = sum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(~0u, incl, o);
                    if (lane >= o) incl += y;
                }
                const int above = incl - sum;
                if (above < kk && kk <= above + sum) {
                    int a = above;
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        if (kk <= a + cnt[e]) {
                            s_prefix = prefix | ((uint32_t)(255 - 8 * lane - e) << shift);
                            s_kk = kk - a;
                            break;
                        }
                        a += cnt[e];
                    }
                }
            }
            __syncthreads();
            prefix = s_prefix;
            kk = s_kk;
        }
    }
    const bool none = c.slots == 0;
    const uint32_t thr = prefix;
    const int k_eq = none ? 0 : kk;

    // ---- ordered emission
    int neq = 0;
    if (!none) {
        int cr = cbase;
        for (int j = j0; j < j1; ++j)
            if ((modality[j] != 0) == (cand_mod != 0)) {
                neq += (cr < n_cand && !is_sink(p, j) && keys[cr] == thr);
                ++cr;
            }
    }
    const int ebase = block_exclusive_scan(neq, scan_buf, &tot);
    // kept(j): a sink, a text key when vision keys are ranked, or a ranked
    // candidate above T, or one of the first k_eq equal to T
    auto scan_kept = [&](auto&& emit) {
        int cr = cbase, er = ebase;
        for (int j = j0; j < j1; ++j) {
            const bool isc = (modality[j] != 0) == (cand_mod != 0);
            bool keep = is_sink(p, j) || (c.vision && modality[j] == 0);
            if (isc) {
                if (!keep && !none && cr < n_cand) {
                    const uint32_t key = keys[cr];
                    if (key > thr) {
                        keep = true;
                    } else if (key == thr) {
                        keep = er < k_eq;
                        ++er;
                    }
                }
                ++cr;
            }
            if (keep) emit(j);
        }
    };
    int nkeep = 0;
    scan_kept([&](int) { ++nkeep; });
    const int kbase = block_exclusive_scan(nkeep, scan_buf, &tot);
    const long long off = s_off;
    {
        int r = kbase;
        scan_kept([&](int j) {
            if (r < len) {
                idx[off + r] = j;
                if (COMPACT) rows[r] = j;
            }
            ++r;
        });
    }
    if (tid == 0 && tot != len) raise_status(status, TGVKV_STATUS_COUNT);
    if (!COMPACT) return;

    __syncthreads();
    constexpr int RPI = 32 / VPR;
    constexpr int UNROLL = 4;
    const int n = min(len, tot);
    const int sub = lane / VPR, vec = lane % VPR;
    const size_t head = (size_t)lg * p.N;
    for (int r0 = warp * RPI * UNROLL; r0 < n; r0 += (kThreads / 32) * RPI * UNROLL) {
        uint4 kr[UNROLL], vr[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int r = r0 + u * RPI + sub;
            if (r < n) {
                const size_t src = (head + rows[r]) * VPR + vec;
                kr[u] = __ldg(k + src);
                vr[u] = __ldg(v + src);
            }
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int r = r0 + u * RPI + sub;
            if (r < n) {
                const size_t dst = (size_t)(off + r) * VPR + vec;
                k_out[dst] = kr[u];
                v_out[dst] = vr[u];
            }
        }
    }
}

template <bool COMPACT, int VPR>
cudaError_t launch_sel_general(const Problem& p, const float* scores, const float* text_scores,
                               const int32_t* budgets, const uint8_t* modality, int64_t* offsets,
                               int32_t* idx, const uint16_t* k, const uint16_t* v, uint16_t* k_out,
                               uint16_t* v_out, long long capacity, uint32_t* status,
                               cudaStream_t stream) {
    auto kern = tpr_select_general_kernel<COMPACT, VPR>;
    const size_t smem = select_general_smem(p, COMPACT);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<p.L * p.H_kv, kThreads, smem, stream>>>(
        p, scores, text_scores, budgets, modality, offsets, idx, reinterpret_cast<const uint4*>(k),
        reinterpret_cast<const uint4*>(v), reinterpret_cast<uint4*>(k_out),
        reinterpret_cast<uint4*>(v_out), capacity, status);
    return cudaGetLastError();
}

// The hot-path kernels cover the vision basis without sinks.
inline bool general_select(const Problem& p) {
    return p.basis == TGVKV_BASIS_ALL || p.keep_first > 0 || p.keep_last > 0 || p.head_budgets;
}

// Warps per CTA of the warp-per-head kernel for p (0: use the CTA-per-head
// kernel): only when there are many heads and eight heads' tables fit in
// 64 KB, so that enough warps share an SM to keep the gather's loads in
// flight (measured on GB300: faster for 1024 heads of 675 keys, slower for
// 1024 heads of 3008 keys at four warps per CTA).
inline int warp_select_warps(const Problem& p) {
    const size_t per_warp = sizeof(uint32_t) * warp_select_words(p);
    if (p.L * p.H_kv < 512) return 0;
    return per_warp * 8 + (size_t)p.N <= 64 * 1024 ? 8 : 0;
}

template <int VPR>
cudaError_t launch_sel_warp(const Problem& p, int nw, const float* scores, const int32_t* budgets,
                            const uint8_t* modality, int64_t* offsets, int32_t* idx,
                            const uint16_t* k, const uint16_t* v, uint16_t* k_out, uint16_t* v_out,
                            long long capacity, uint32_t* status, cudaStream_t stream) {
    auto kern = tpr_select_warp_kernel<VPR>;
    const size_t smem = (((size_t)p.N + 15) & ~size_t(15)) + sizeof(uint32_t) * warp_select_words(p) * nw;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int heads = p.L * p.H_kv;
    // a programmatic dependent of the kernel before (the score kernel on the evict path)
    return launch_dependent(kern, dim3(2 * ((heads + nw - 1) / nw)), dim3(nw * 32), smem, stream, p,
                            scores, budgets, modality, offsets, idx, reinterpret_cast<const uint4*>(k),
                            reinterpret_cast<const uint4*>(v), reinterpret_cast<uint4*>(k_out),
                            reinterpret_cast<uint4*>(v_out), capacity, status);
}

template <bool COMPACT, int VPR>
cudaError_t launch_sel(const Problem& p, const float* scores, const int32_t* budgets,
                       const uint8_t* modality, int64_t* offsets, int32_t* idx,
                       const uint16_t* k, const uint16_t* v, uint16_t* k_out, uint16_t* v_out,
                       long long capacity, uint32_t* status, cudaStream_t stream) {
    auto kern = tpr_select_kernel<COMPACT, VPR>;
    const size_t smem = select_smem(p, COMPACT);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid(p.L * p.H_kv * (COMPACT ? 2 : 1));
    if (COMPACT)   // a programmatic dependent of the kernel before (the score kernel on the evict path)
        return launch_dependent(kern, grid, dim3(kThreads), smem, stream, p, scores, budgets, modality,
                                offsets, idx, reinterpret_cast<const uint4*>(k),
                                reinterpret_cast<const uint4*>(v), reinterpret_cast<uint4*>(k_out),
                                reinterpret_cast<uint4*>(v_out), capacity, status);
    kern<<<grid, kThreads, smem, stream>>>(
        p, scores, budgets, modality, offsets, idx,
        reinterpret_cast<const uint4*>(k),
        reinterpret_cast<const uint4*>(v), reinterpret_cast<uint4*>(k_out),
        reinterpret_cast<uint4*>(v_out), capacity, status);
    return cudaGetLastError();
}

// The select-only form writes no rows; its index capacity is the caller's
// (tgvkv_retained_rows for sets of a split the budget call made).
constexpr long long kNoCapacity = 0x7FFFFFFFFFFFFFFFLL;

// Select only; a set that would end past `capacity` indices writes none.
cudaError_t launch_select_cap(const Problem& p, const float* scores, const float* text_scores,
                              const int32_t* budgets, const uint8_t* modality, int64_t* offsets,
                              int32_t* idx, long long capacity, uint32_t* status,
                              cudaStream_t stream) {
    if (general_select(p))
        return launch_sel_general<false, 16>(p, scores, text_scores, budgets, modality, offsets,
                                             idx, nullptr, nullptr, nullptr, nullptr, capacity,
                                             status, stream);
    return launch_sel<false, 16>(p, scores, budgets, modality, offsets, idx, nullptr, nullptr, nullptr,
                                 nullptr, capacity, status, stream);
}

}  // namespace

cudaError_t launch_select(const Problem& p, const float* scores, const float* text_scores,
                          const int32_t* budgets, const uint8_t* modality, int64_t* offsets,
                          int32_t* idx, uint32_t* status, cudaStream_t stream) {
    return launch_select_cap(p, scores, text_scores, budgets, modality, offsets, idx, kNoCapacity,
                             status, stream);
}

int select_compact_launches(const Problem& p) {
    if (general_select(p)) return select_general_smem(p, true) > kFusedSmemLimit ? 2 : 1;
    return warp_select_warps(p) == 0 && select_smem(p, true) > kFusedSmemLimit ? 2 : 1;
}

cudaError_t launch_select_compact(const Problem& p, const float* scores, const float* text_scores,
                                  const int32_t* budgets, const uint8_t* modality,
                                  int64_t* offsets, int32_t* idx, const uint16_t* k,
                                  const uint16_t* v, uint16_t* k_out, uint16_t* v_out,
                                  long long capacity_rows, uint32_t* status, cudaStream_t stream) {
    if (general_select(p)) {
        if (select_general_smem(p, true) > kFusedSmemLimit) {
            cudaError_t e = launch_select_cap(p, scores, text_scores, budgets, modality, offsets,
                                              idx, capacity_rows, status, stream);
            if (e != cudaSuccess) return e;
            return launch_compact(p, k, v, offsets, idx, k_out, v_out, capacity_rows, status,
                                  stream, /*whole_sets=*/true);
        }
        if (p.d == 64)
            return launch_sel_general<true, 8>(p, scores, text_scores, budgets, modality, offsets,
                                               idx, k, v, k_out, v_out, capacity_rows, status,
                                               stream);
        return launch_sel_general<true, 16>(p, scores, text_scores, budgets, modality, offsets, idx,
                                            k, v, k_out, v_out, capacity_rows, status, stream);
    }
    if (const int nw = warp_select_warps(p)) {
        if (p.d == 64)
            return launch_sel_warp<8>(p, nw, scores, budgets, modality, offsets, idx, k, v, k_out,
                                      v_out, capacity_rows, status, stream);
        return launch_sel_warp<16>(p, nw, scores, budgets, modality, offsets, idx, k, v, k_out,
                                   v_out, capacity_rows, status, stream);
    }
    if (select_smem(p, true) > kFusedSmemLimit) {
        cudaError_t e = launch_select_cap(p, scores, nullptr, budgets, modality, offsets, idx,
                                          capacity_rows, status, stream);
        if (e != cudaSuccess) return e;
        return launch_compact(p, k, v, offsets, idx, k_out, v_out, capacity_rows, status, stream,
                              /*whole_sets=*/true);
    }
    if (p.d == 64)
        return launch_sel<true, 8>(p, scores, budgets, modality, offsets, idx, k, v, k_out, v_out,
                                   capacity_rows, status, stream);
    return launch_sel<true, 16>(p, scores, budgets, modality, offsets, idx, k, v, k_out, v_out,
                                capacity_rows, status, stream);
}

}  // namespace tgvkv
