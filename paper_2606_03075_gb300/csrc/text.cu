// Eq. 7: the derived text weights w~ of one layer from the Eq. 9 text scores.
//
// Both equations read the same text-text slice of the causal attention: the
// Eq. 9 score of text key t is the column sum over the query rows of
// A[i, t], averaged over the G query heads of a KV head.  Eq. 7 takes, for the
// query row j (a text token at position p_j), the column p_j summed over the
// rows at or after j -- rows before j see p_j as 0 through the causal mask --
// averaged over all H_q heads and divided by the n_win - j rows:
//   w_{l,j} = sum_g text_scores[l][g][rank(p_j)] / (H_kv * (n_win - j))
// (the mean over the G heads of a group times G, over H_q = G * H_kv heads).
// Then w~_{l,j} = w_{l,j} / sum_j' w_{l,j'}.  One CTA per layer; the sum runs
// in a fixed order, so the weights are reproducible.
#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kThreads = 256;
constexpr int kWords = kMaxN / 32;

__global__ void __launch_bounds__(kThreads)
eq7_weights_kernel(Problem p, const float* __restrict__ text_scores,
                   const uint8_t* __restrict__ modality, const int32_t* __restrict__ text_pos,
                   float* __restrict__ weights, uint32_t* __restrict__ status) {
    __shared__ uint32_t word[kWords];     // text bit of each position
    __shared__ int before[kWords];        // text positions before each 32-position word
    __shared__ int warp_sum[kThreads / 32];
    __shared__ float part[kThreads];
    const int l = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nwords = (p.N + 31) / 32;
    for (int wd = warp; wd < nwords; wd += kThreads / 32) {
        const int j = wd * 32 + lane;
        const unsigned m = __ballot_sync(~0u, j < p.N && modality[j] == 0);
        if (lane == 0) word[wd] = m;
    }
    __syncthreads();
    // exclusive scan of the per-word text counts: contiguous words per thread
    const int wper = (nwords + kThreads - 1) / kThreads;
    const int w0 = min(nwords, tid * wper), w1 = min(nwords, w0 + wper);
    int cnt = 0;
    for (int wd = w0; wd < w1; ++wd) cnt += __popc(word[wd]);
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(~0u, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_sum[warp] = incl;
    __syncthreads();
    int run = incl - cnt;
    for (int x = 0; x < warp; ++x) run += warp_sum[x];
    for (int wd = w0; wd < w1; ++wd) {
        before[wd] = run;
        run += __popc(word[wd]);
    }
    __syncthreads();

    // raw weights of this thread's contiguous range of rows
    const int per = (p.n_win + kThreads - 1) / kThreads;
    const int j0 = min(p.n_win, tid * per), j1 = min(p.n_win, j0 + per);
    float* wl = weights + (size_t)l * p.n_win;
    const float* ts = text_scores + (size_t)l * p.H_kv * p.N_t;
    float acc = 0.f;
    for (int j = j0; j < j1; ++j) {
        const int pos = text_pos[j];
        float wj = 0.f;
        if (pos < 0 || pos >= p.N || ((word[pos >> 5] >> (pos & 31)) & 1u) == 0u) {
            raise_status(status, TGVKV_STATUS_TEXT_POS);
        } else {
            const int t = before[pos >> 5] + __popc(word[pos >> 5] & ((1u << (pos & 31)) - 1u));
            float sum = 0.f;
            for (int g = 0; g < p.H_kv; ++g) sum += ts[(size_t)g * p.N_t + t];
            wj = sum / ((float)p.H_kv * (float)(p.n_win - j));
        }
        wl[j] = wj;
        acc += wj;
    }
    // the layer's sum, in a fixed order: thread ranges, then a fixed tree
    part[tid] = acc;
    __syncthreads();
    for (int o = kThreads / 2; o > 0; o >>= 1) {
        if (tid < o) part[tid] += part[tid + o];
        __syncthreads();
    }
    const float total = part[0];
    for (int j = j0; j < j1; ++j) wl[j] = total > 0.f ? wl[j] / total : 0.f;
}

}  // namespace

cudaError_t launch_eq7_weights(const Problem& p, const float* text_scores, const uint8_t* modality,
                               const int32_t* text_pos, float* weights, uint32_t* status,
                               cudaStream_t stream) {
    if (p.n_win == 0) return cudaSuccess;
    eq7_weights_kernel<<<p.L, kThreads, 0, stream>>>(p, text_scores, modality, text_pos, weights,
                                                     status);
    return cudaGetLastError();
}

}  // namespace tgvkv
