// TPR retention (Eq. 10, case b_l > N_t, vision budget b_l): one CTA per
// (layer, KV head) keeps every text position and the b_l vision positions of
// highest score, ties to the lower position, and writes them in ascending
// position order.
//
// Selection: the scores are mapped to order-preserving 32-bit keys in shared
// memory; an MSB-first radix select (four 8-bit digits) finds the key T of the
// b_l-th largest score and how many keys equal to T are still needed (k_eq).
// A vision key is kept iff key > T, or key == T and it is among the first k_eq
// such keys in position order.  One ordered pass over the positions then
// emits text and kept vision positions through block prefix sums.
#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kThreads = 1024;

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
        const int v = (lane < (int)(blockDim.x >> 5)) ? buf[lane] : 0;
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

__global__ void __launch_bounds__(kThreads)
tpr_select_kernel(Problem p, const float* __restrict__ scores, const int32_t* __restrict__ budgets,
                  const uint8_t* __restrict__ modality, int64_t* __restrict__ offsets,
                  int32_t* __restrict__ idx, uint32_t* __restrict__ status) {
    extern __shared__ uint32_t keys[];  // [N_v]
    __shared__ int hist[256];
    __shared__ int scan_buf[33];
    __shared__ uint32_t s_prefix;
    __shared__ int s_kk;
    __shared__ long long s_off;

    const int lg = blockIdx.x, l = lg / p.H_kv, g = lg % p.H_kv;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    int b = budgets[l];
    if (b < 0 || b > p.N_v) {
        if (tid == 0) raise_status(status, TGVKV_STATUS_BUDGET);
        b = b < 0 ? 0 : p.N_v;
    }
    const int len = p.N_t + b;
    if (tid == 0) {
        long long off = 0;
        for (int m = 0; m < l; ++m) {
            int bm = budgets[m];
            bm = bm < 0 ? 0 : (bm > p.N_v ? p.N_v : bm);
            off += (long long)p.H_kv * (p.N_t + bm);
        }
        off += (long long)g * len;
        s_off = off;
        offsets[lg] = off;
        if (lg == p.L * p.H_kv - 1) offsets[lg + 1] = off + len;
    }
    const float* sc = scores + (size_t)lg * p.N_v;
    for (int v = tid; v < p.N_v; v += kThreads) keys[v] = float_order_key(sc[v]);
    __syncthreads();

    // ---- radix select of the b-th largest key
    uint32_t prefix = 0;
    int kk = b;
    if (b > 0) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            if (tid < 256) hist[tid] = 0;
            __syncthreads();
            const uint32_t hi_mask = (shift == 24) ? 0u : (0xFFFFFFFFu << (shift + 8));
            for (int v = tid; v < p.N_v; v += kThreads) {
                const uint32_t key = keys[v];
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

    // ---- ordered emission: text positions and kept vision positions
    const long long off = s_off;
    int vis_run = 0, eq_run = 0, keep_run = 0;
    for (int base = 0; base < p.N; base += kThreads) {
        const int j = base + tid;
        const int is_vis = (j < p.N && modality[j] != 0) ? 1 : 0;
        int tot;
        const int vr = vis_run + block_exclusive_scan(is_vis, scan_buf, &tot);
        vis_run += tot;
        int is_eq = 0, is_gt = 0;
        if (is_vis && vr < p.N_v) {
            const uint32_t key = keys[vr];
            is_gt = key > thr;
            is_eq = key == thr;
        }
        const int er = eq_run + block_exclusive_scan(is_eq, scan_buf, &tot);
        eq_run += tot;
        const int keep = (j < p.N) && (!is_vis || (!none && (is_gt || (is_eq && er < k_eq))));
        const int kr = keep_run + block_exclusive_scan(keep, scan_buf, &tot);
        keep_run += tot;
        if (keep && kr < len) idx[off + kr] = j;
    }
    if (tid == 0 && keep_run != len) raise_status(status, TGVKV_STATUS_COUNT);
}

}  // namespace

cudaError_t launch_select(const Problem& p, const float* scores, const int32_t* budgets,
                          const uint8_t* modality, int64_t* offsets, int32_t* idx,
                          uint32_t* status, cudaStream_t stream) {
    const size_t smem = sizeof(uint32_t) * (size_t)p.N_v;
    cudaError_t e = cudaFuncSetAttribute(tpr_select_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    tpr_select_kernel<<<p.L * p.H_kv, kThreads, smem, stream>>>(p, scores, budgets, modality,
                                                                offsets, idx, status);
    return cudaGetLastError();
}

}  // namespace tgvkv
