// TVB layer budgets (Eq. 5, x = TV): one CTA splits B_V vision rows over the
// layers in proportion to the per-layer text-vision attention sums.
//
// Integer rounding: b_l = floor(q_l) with q_l = B * S_l / sum S, plus one unit
// for each of the B - sum floor(q) layers with the largest fractional part
// (ties: lower layer).  Layers whose budget exceeds N_v are capped and the rest
// is split again over the others.  Quotients are computed in double with
// explicitly rounded operations (no contraction), and the denominator is
// summed in ascending layer order, so the integers are reproducible.
#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kThreads = 1024;

__global__ void __launch_bounds__(kThreads)
tvb_budget_kernel(const float* __restrict__ stat, int L, long long total, int cap,
                  int32_t* __restrict__ budgets, uint32_t* __restrict__ status) {
    __shared__ double frac[kMaxL];
    __shared__ long long base[kMaxL];
    __shared__ unsigned char active[kMaxL];
    __shared__ int result[kMaxL];
    __shared__ double denom;
    __shared__ long long remaining;
    __shared__ long long leftover;
    __shared__ int n_active, any_over;

    const int tid = threadIdx.x;
    for (int l = tid; l < L; l += kThreads) {
        active[l] = 1;
        result[l] = 0;
    }
    if (tid == 0) {
        remaining = total;
        n_active = L;
    }
    __syncthreads();
    for (int round = 0; round <= L; ++round) {
        if (tid == 0) {
            double s = 0.0;
            for (int l = 0; l < L; ++l)
                if (active[l]) s = __dadd_rn(s, (double)stat[l]);
            denom = s;
            any_over = 0;
        }
        __syncthreads();
        const double rem = (double)remaining;
        for (int l = tid; l < L; l += kThreads) {
            if (!active[l]) continue;
            const double qv = denom > 0.0 ? __ddiv_rn(__dmul_rn(rem, (double)stat[l]), denom)
                                          : __ddiv_rn(rem, (double)n_active);
            const double fl = floor(qv);
            base[l] = (long long)fl;
            frac[l] = __dsub_rn(qv, fl);
        }
        __syncthreads();
        // leftover units: one each to the layers of rank < leftover by
        // (fraction desc, layer asc)
        if (tid == 0) {
            long long floors = 0;
            for (int l = 0; l < L; ++l)
                if (active[l]) floors += base[l];
            leftover = remaining - floors;
        }
        __syncthreads();
        for (int l = tid; l < L; l += kThreads) {
            if (!active[l]) continue;
            long long rank = 0;
            for (int m = 0; m < L; ++m) {
                if (!active[m] || m == l) continue;
                if (frac[m] > frac[l] || (frac[m] == frac[l] && m < l)) ++rank;
            }
            long long b = base[l] + (rank < leftover ? 1 : 0);
            base[l] = b;
            if (b > cap) any_over = 1;
        }
        __syncthreads();
        if (!any_over) {
            for (int l = tid; l < L; l += kThreads)
                if (active[l]) result[l] = (int)base[l];
            break;
        }
        __syncthreads();
        if (tid == 0) {
            for (int l = 0; l < L; ++l) {
                if (active[l] && base[l] > cap) {
                    active[l] = 0;
                    result[l] = cap;
                    remaining -= cap;
                    --n_active;
                }
            }
            if (n_active == 0 && remaining != 0) raise_status(status, TGVKV_STATUS_BUDGET);
        }
        __syncthreads();
        if (n_active == 0) break;
    }
    __syncthreads();
    for (int l = tid; l < L; l += kThreads) budgets[l] = result[l];
}

}  // namespace

cudaError_t launch_budget(const Problem& p, const float* tvb_stat, long long total,
                          int32_t* budgets, uint32_t* status, cudaStream_t stream) {
    tvb_budget_kernel<<<1, kThreads, 0, stream>>>(tvb_stat, p.L, total, p.N_v, budgets, status);
    return cudaGetLastError();
}

}  // namespace tgvkv
