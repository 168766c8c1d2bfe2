// Host-side launchers of the TGV-KV kernels (one per step).  All of them are
// asynchronous on `stream` and assume the arguments were validated by the
// C-ABI layer.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace tgvkv {

// Launch `kern` as a programmatic dependent of the kernel before it on
// `stream` (see griddep_wait): its CTAs may be scheduled while that kernel
// finishes, and must call griddep_wait before reading what it wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t stream, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

// TWR scores + TVB statistic (score_tc.cu).  The completion counters in the
// workspace must be zero on entry; the kernel leaves them zero.  When
// `budgets` is not null, the CTA that finishes last also splits
// `budget_total` over the layers (Eq. 5) into budgets[L].
cudaError_t launch_score(const Problem& p, const uint16_t* q, const uint16_t* k,
                         const uint8_t* modality, const int32_t* text_pos, const float* w,
                         float* scores, float* tvb_stat, char* ws, const WsLayout& lay,
                         long long budget_total, int32_t* budgets, cudaStream_t stream);

// TVB split of `total` (budget.cu); the cap is N_v (vision basis) or N.
cudaError_t launch_budget(const Problem& p, const float* tvb_stat, long long total,
                          int32_t* budgets, uint32_t* status, cudaStream_t stream);

// TPR selection (select.cu).  text_scores (Eq. 9) is read only under the
// all-token basis for layers with b_l <= N_t.
cudaError_t launch_select(const Problem& p, const float* scores, const float* text_scores,
                          const int32_t* budgets, const uint8_t* modality, int64_t* offsets,
                          int32_t* idx, uint32_t* status, cudaStream_t stream);

// select + gather fused (tgvkv_evict): one CTA per (layer, KV head) selects
// its set and gathers its rows; falls back to the separate select and compact
// kernels when the keys and retained rows of a head do not fit in shared
// memory.
cudaError_t launch_select_compact(const Problem& p, const float* scores, const float* text_scores,
                                  const int32_t* budgets, const uint8_t* modality,
                                  int64_t* offsets, int32_t* idx, const uint16_t* k,
                                  const uint16_t* v, uint16_t* k_out, uint16_t* v_out,
                                  long long capacity_rows, uint32_t* status, cudaStream_t stream);

// Eq. 7 weights from the Eq. 9 text scores (text.cu): weights[l][j] for the
// query rows, L1-normalised per layer.
cudaError_t launch_eq7_weights(const Problem& p, const float* text_scores, const uint8_t* modality,
                               const int32_t* text_pos, float* weights, uint32_t* status,
                               cudaStream_t stream);

// Decode over the compacted cache (decode.cu): out[l][h][:] for one new token
// (two kernels: the row streams, then the merge of the sets they split).  Rows
// from capacity_rows on are never read.
cudaError_t launch_decode(const Problem& p, const uint16_t* q, const uint16_t* k_rows,
                          const uint16_t* v_rows, long long capacity_rows, const int64_t* offsets,
                          float* out, float* part, uint32_t* status, cudaStream_t stream);
int decode_launches(const Problem& p);

// Kernels launch_score / launch_select_compact launch for p.
int score_launches(const Problem& p);
int select_compact_launches(const Problem& p);

// Causal prefill attention over every token (prefill.cu), which also writes
// the eviction step's query rows (q_text) and their (m, Z, vision mass).
cudaError_t launch_prefill(const Problem& p, const uint16_t* q, const uint16_t* k,
                           const uint16_t* v, const uint8_t* modality, const int32_t* text_pos,
                           uint16_t* o, uint16_t* q_text, float* row_stats, uint32_t* status,
                           cudaStream_t stream);

// TMA map of a bf16 [rows][d] tensor with boxes of 64 x box_rows, 128-byte
// swizzle (score_tc.cu), and the SM count of the current device.
bool make_tile_map(CUtensorMap* map, const void* base, uint64_t rows, int d, uint32_t box_rows);
int device_sm_count();

// One CTA that waits, with the library's bounded wait, on an mbarrier nothing
// arrives at; the wait runs out and sets TGVKV_STATUS_TIMEOUT (selftest.cu).
cudaError_t launch_wait_timeout(uint32_t* status, cudaStream_t stream);

// Compaction (compact.cu).  Rows from capacity_rows on are never written;
// with whole_sets, neither is any row of a set that ends past capacity_rows.
cudaError_t launch_compact(const Problem& p, const uint16_t* k, const uint16_t* v,
                           const int64_t* offsets, const int32_t* idx, uint16_t* k_out,
                           uint16_t* v_out, long long capacity_rows, uint32_t* status,
                           cudaStream_t stream, bool whole_sets = false);

}  // namespace tgvkv
