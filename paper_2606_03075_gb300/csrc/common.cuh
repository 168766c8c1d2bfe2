// Device-side helpers shared by the TGV-KV kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "tgvkv.h"

namespace tgvkv {

// Problem as the kernels see it.  Built on the host from tgvkv_desc.
struct Problem {
    int L, H_q, H_kv, G, d, N, N_v, N_t, n_win;
    int R;                 // query rows per KV head: G * n_win
    int T;                 // 128-row tiles per KV head: ceil(R / 128)
    float scale_log2;      // softmax_scale * log2(e): logits in base-2 units
    long long w_stride;    // floats between the weight rows of two layers
};

// Workspace layout (byte offsets into the caller's buffer).
struct WsLayout {
    size_t status;      // uint32 status word
    size_t tickets;     // uint32 [L*H_kv + L]: completion counters
    size_t stat_part;   // float [L*H_kv*T]: TV mass of one row tile
    size_t stat_head;   // float [L*H_kv]: TV mass of one KV head
    size_t score_part;  // float [L*H_kv*T*N_v]: scores of one row tile (T > 1)
    size_t total;
};

constexpr int kMaxN = 32768;     // key positions per head (the per-CTA tile maps)
constexpr int kMaxNv = 49152;    // vision keys held in shared memory by select
constexpr int kMaxL = 1024;      // layers handled by the budget kernel

__device__ __forceinline__ void raise_status(uint32_t* status, uint32_t bits) {
    atomicOr(status, bits);
}

// 2^x with the MUFU.EX2 unit (PTX ex2.approx.ftz.f32; ex2(-inf) = +0).
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// log2(x) with the MUFU.LG2 unit (PTX lg2.approx.ftz.f32; lg2(0) = -inf).
__device__ __forceinline__ float fast_log2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---- Ampere-style async copy and warp MMA (used by the streaming score kernel)
__device__ __forceinline__ void cp_async_16(uint32_t saddr, const void* gptr) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(saddr), "l"(gptr));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D += A * B, m16n8k16, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Order-preserving map of an fp32 value to uint32 (larger float -> larger key).
__device__ __forceinline__ uint32_t float_order_key(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

}  // namespace tgvkv
