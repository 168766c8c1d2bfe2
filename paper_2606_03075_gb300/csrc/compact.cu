// Compaction: gather the K and V rows of every retained position into the
// dense output cache (bit copies).  Output row r of set (l, g) comes from row
// idx[r] of head (l, g).  The grid runs over output rows; each warp copies a
// run of consecutive rows with 16-byte vector loads and stores (a row of d
// bf16 values is d/8 vectors), issuing all its loads before its stores.
#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kThreads = 256;
constexpr int kIter = 4;

template <int VPR>  // 16-byte vectors per row: d * 2 / 16
__global__ void __launch_bounds__(kThreads)
compact_kernel(Problem p, const uint4* __restrict__ k, const uint4* __restrict__ v,
               const int64_t* __restrict__ offsets, const int32_t* __restrict__ idx,
               uint4* __restrict__ k_out, uint4* __restrict__ v_out, long long capacity,
               int whole_sets, uint32_t* __restrict__ status) {
    constexpr int RPI = 32 / VPR;                 // rows per warp per iteration
    constexpr int ROWS_PER_WARP = RPI * kIter;
    constexpr int ROWS_PER_CTA = ROWS_PER_WARP * (kThreads / 32);
    const int n_heads = p.L * p.H_kv;
    long long total = offsets[n_heads];
    if (total < 0 || total > capacity) {
        // a CSR that does not fit the output: write the rows that do
        if (blockIdx.x == 0 && threadIdx.x == 0) raise_status(status, TGVKV_STATUS_INDEX);
        total = total < 0 ? 0 : capacity;
    }
    // the sets must lie in order (every access below stays in bounds either way)
    for (int i = blockIdx.x * kThreads + threadIdx.x; i < n_heads; i += gridDim.x * kThreads)
        if (offsets[i + 1] < offsets[i]) raise_status(status, TGVKV_STATUS_INDEX);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long r0 = (long long)blockIdx.x * ROWS_PER_CTA + (long long)warp * ROWS_PER_WARP;
    if (r0 >= total) return;
    const int sub = lane / VPR, vec = lane % VPR;

    // head of row r0: offsets[lo] <= r0 < offsets[lo + 1]
    int lo = 0, hi = n_heads;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (offsets[mid] <= r0) lo = mid; else hi = mid;
    }
    int lg = lo;

    uint4 kr[kIter], vr[kIter];
    long long rows[kIter];
    bool ok[kIter];
#pragma unroll
    for (int it = 0; it < kIter; ++it) {
        const long long r = r0 + it * RPI + sub;
        rows[it] = r;
        ok[it] = r < total;
        if (ok[it]) {
            while (offsets[lg + 1] <= r) ++lg;
            if (whole_sets && offsets[lg + 1] > capacity) ok[it] = false;   // its set does not fit
        }
        if (ok[it]) {
            const int src = idx[r];
            if (src < 0 || src >= p.N) {
                raise_status(status, TGVKV_STATUS_INDEX);
                ok[it] = false;
            } else {
                const size_t s = ((size_t)lg * p.N + src) * VPR + vec;
                kr[it] = __ldg(k + s);
                vr[it] = __ldg(v + s);
            }
        }
    }
#pragma unroll
    for (int it = 0; it < kIter; ++it) {
        if (ok[it]) {
            k_out[rows[it] * VPR + vec] = kr[it];
            v_out[rows[it] * VPR + vec] = vr[it];
        }
    }
}

template <int VPR>
cudaError_t launch_compact_t(const Problem& p, const uint16_t* k, const uint16_t* v,
                             const int64_t* offsets, const int32_t* idx, uint16_t* k_out,
                             uint16_t* v_out, long long capacity_rows, bool whole_sets,
                             uint32_t* status, cudaStream_t stream) {
    constexpr int ROWS_PER_CTA = (32 / VPR) * kIter * (kThreads / 32);
    const long long blocks = (capacity_rows + ROWS_PER_CTA - 1) / ROWS_PER_CTA;
    if (blocks == 0) return cudaSuccess;
    compact_kernel<VPR><<<(unsigned)blocks, kThreads, 0, stream>>>(
        p, reinterpret_cast<const uint4*>(k), reinterpret_cast<const uint4*>(v), offsets, idx,
        reinterpret_cast<uint4*>(k_out), reinterpret_cast<uint4*>(v_out), capacity_rows,
        whole_sets ? 1 : 0, status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_compact(const Problem& p, const uint16_t* k, const uint16_t* v,
                           const int64_t* offsets, const int32_t* idx, uint16_t* k_out,
                           uint16_t* v_out, long long capacity_rows, uint32_t* status,
                           cudaStream_t stream, bool whole_sets) {
    if (p.d == 64)
        return launch_compact_t<8>(p, k, v, offsets, idx, k_out, v_out, capacity_rows, whole_sets,
                                   status, stream);
    return launch_compact_t<16>(p, k, v, offsets, idx, k_out, v_out, capacity_rows, whole_sets,
                                status, stream);
}

}  // namespace tgvkv
