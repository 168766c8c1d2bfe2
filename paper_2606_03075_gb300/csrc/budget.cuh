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

// tvb_budget_block for at most 32 units, by one warp (lane l = unit l, every
// lane of the warp calling): the same double operations in the same order --
// the denominator summed over the active units in unit order, the quotient
// rounded multiply then rounded divide, the fractional part's bit pattern
// ranked (fraction desc, unit asc) -- so the same integers, with warp
// shuffles in place of the block's shared scratch and barriers.  stat: the
// statistic of unit `lane` (ignored when uniform).
__device__ __forceinline__ void tvb_budget_warp(float stat, int L, long long total, int cap,
                                                int32_t* budgets, uint32_t* status, bool uniform,
                                                int lane) {
    const bool has = lane < L;
    const double st = (has && !uniform) ? (double)stat : 0.0;
    bool active = has;
    int result = 0;
    long long remaining = total;
    int n_active = L;
    for (int round = 0; round <= L; ++round) {
        const uint32_t act = __ballot_sync(~0u, active);
        double den = 0.0;
        for (int m = 0; m < L; ++m) {
            const double sm = __shfl_sync(~0u, st, m);
            if ((act >> m) & 1u) den = __dadd_rn(den, sm);
        }
        const double rem = (double)remaining;
        long long base = 0;
        unsigned long long frac = 0;
        if (active) {
            const double qv = den > 0.0 ? __ddiv_rn(__dmul_rn(rem, st), den)
                                        : __ddiv_rn(rem, (double)n_active);
            const double fl = floor(qv);
            base = (long long)fl;
            frac = (unsigned long long)__double_as_longlong(__dsub_rn(qv, fl));
        }
        long long floors = base;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) floors += __shfl_xor_sync(~0u, floors, o);
        const long long leftover = remaining - floors;
        long long rank = 0;
        for (int m = 0; m < L; ++m) {
            const unsigned long long fm = __shfl_sync(~0u, frac, m);
            if (active && ((act >> m) & 1u) && m != lane && (fm > frac || (fm == frac && m < lane)))
                ++rank;
        }
        const long long v = base + (rank < leftover ? 1 : 0);
        const uint32_t over = __ballot_sync(~0u, active && v > cap);
        if (over == 0u) {
            if (active) result = (int)v;
            break;
        }
        if ((over >> lane) & 1u) {
            active = false;
            result = cap;
        }
        const int n_over = __popc(over);
        remaining -= (long long)cap * n_over;
        n_active -= n_over;
        if (n_active == 0 && remaining != 0 && lane == 0) raise_status(status, TGVKV_STATUS_BUDGET);
        if (n_active == 0) break;
    }
    if (has && budgets) budgets[lane] = result;
}

}  // namespace tgvkv
