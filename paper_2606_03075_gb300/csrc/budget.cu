// TVB layer budgets (Eq. 5, x = TV): the standalone tgvkv_budget kernel, one
// CTA running the block-wide split of budget.cuh.
#include "budget.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kThreads = 512;

__global__ void __launch_bounds__(kThreads)
tvb_budget_kernel(const float* __restrict__ stat, int L, long long total, int cap, int uniform,
                  int32_t* __restrict__ budgets, uint32_t* __restrict__ status) {
    __shared__ BudgetScratch scratch;
    tvb_budget_block(stat, L, total, cap, budgets, status, scratch, uniform != 0);
}

}  // namespace

cudaError_t launch_budget(const Problem& p, const float* tvb_stat, long long total,
                          int32_t* budgets, uint32_t* status, cudaStream_t stream) {
    const int cap = p.basis == TGVKV_BASIS_ALL ? p.N : p.N_v;
    const int units = p.head_budgets ? p.L * p.H_kv : p.L;
    tvb_budget_kernel<<<1, kThreads, 0, stream>>>(tvb_stat, units, total, cap,
                                                  p.budget_stat == TGVKV_STAT_UNIFORM, budgets, status);
    return cudaGetLastError();
}

}  // namespace tgvkv
