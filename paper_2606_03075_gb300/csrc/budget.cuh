// TVB layer budgets (Eq. 5, x = TV) as a block-wide device routine, used by
// the standalone budget kernel and by the last CTA of the fused score kernel.
//
// Splits `total` vision rows over L layers in proportion to stat[l]:
// b_l = floor(q_l), q_l = remaining * S_l / sum S, plus one leftover unit for
// each of the layers with the largest fractional parts (ties: lower layer).
// Layers above `cap` (= N_v) are capped and the rest is split again over the
// other layers; an all-zero statistic splits uniformly.  The quotients use
// explicitly rounded double operations (no contraction) and the denominator
// is summed in ascending layer order, so the integers are reproducible.
#pragma once

#include "common.cuh"

namespace tgvkv {

struct BudgetScratch {
    double stat[kMaxL];
    unsigned long long frac[kMaxL];   // bit pattern of the fractional part (order-preserving, >= 0)
    long long base[kMaxL];
    int result[kMaxL];
    unsigned char active[kMaxL];
    double denom;
    long long remaining, leftover;
    int n_active, any_over;
};

// Every thread of the block must call this (it contains __syncthreads); every
// block that calls it with the same statistic gets the same integers.
// `stat` is read once into shared memory with L2-coherent loads.  When
// `budgets` is null the result stays in b.result.  `uniform` ignores the
// statistic (the uniform budgeting of Table 1a: an all-zero statistic).
__device__ __forceinline__ void tvb_budget_block(const float* stat, int L, long long total, int cap,
                                                 int32_t* budgets, uint32_t* status,
                                                 BudgetScratch& b, bool uniform = false) {
    const int tid = threadIdx.x, nt = blockDim.x;
    for (int l = tid; l < L; l += nt) {
        b.stat[l] = uniform ? 0.0 : (double)__ldcg(stat + l);
        b.active[l] = 1;
        b.result[l] = 0;
    }
    if (tid == 0) {
        b.remaining = total;
        b.n_active = L;
    }
    __syncthreads();
    for (int round = 0; round <= L; ++round) {
        if (tid == 0) {
            double s = 0.0;
            for (int l = 0; l < L; ++l)
                if (b.active[l]) s = __dadd_rn(s, b.stat[l]);
            b.denom = s;
            b.any_over = 0;
        }
        __syncthreads();
        const double rem = (double)b.remaining;
        const double den = b.denom;
        for (int l = tid; l < L; l += nt) {
            if (!b.active[l]) continue;
            const double qv = den > 0.0 ? __ddiv_rn(__dmul_rn(rem, b.stat[l]), den)
                                        : __ddiv_rn(rem, (double)b.n_active);
            const double fl = floor(qv);
            b.base[l] = (long long)fl;
            b.frac[l] = (unsigned long long)__double_as_longlong(__dsub_rn(qv, fl));
        }
        __syncthreads();
        if (tid == 0) {
            long long floors = 0;
            for (int l = 0; l < L; ++l)
                if (b.active[l]) floors += b.base[l];
            b.leftover = b.remaining - floors;
        }
        __syncthreads();
        // one leftover unit to each layer of rank < leftover by (fraction desc, layer asc)
        for (int l = tid; l < L; l += nt) {
            if (!b.active[l]) continue;
            long long rank = 0;
            const unsigned long long f = b.frac[l];
            for (int m = 0; m < L; ++m) {
                if (!b.active[m] || m == l) continue;
                if (b.frac[m] > f || (b.frac[m] == f && m < l)) ++rank;
            }
            const long long v = b.base[l] + (rank < b.leftover ? 1 : 0);
            b.base[l] = v;
            if (v > cap) b.any_over = 1;
        }
        __syncthreads();
        if (!b.any_over) {
            for (int l = tid; l < L; l += nt)
                if (b.active[l]) b.result[l] = (int)b.base[l];
            break;
        }
        __syncthreads();
        if (tid == 0) {
            for (int l = 0; l < L; ++l) {
                if (b.active[l] && b.base[l] > cap) {
                    b.active[l] = 0;
                    b.result[l] = cap;
                    b.remaining -= cap;
                    --b.n_active;
                }
            }
            if (b.n_active == 0 && b.remaining != 0) raise_status(status, TGVKV_STATUS_BUDGET);
        }
        __syncthreads();
        if (b.n_active == 0) break;
    }
    __syncthreads();
    if (budgets)
        for (int l = tid; l < L; l += nt) budgets[l] = b.result[l];
}

}  // namespace tgvkv
