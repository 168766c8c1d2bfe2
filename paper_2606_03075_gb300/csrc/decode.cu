// Decode over the compacted cache (the consumer of the eviction step; the
// decode phase of Section 3.1): the new token's query of head h attends to the
// retained rows of KV head g = h / G,
//   o[l][h] = sum_r softmax_r(scale * <q, k_r>) v_r  over the rows r of set (l, g).
// A set without rows gives 0.
//
// One CTA per (layer, KV head, row split, head batch): the G query heads of a
// KV head share every K/V row they read (GQA), at most GB heads per CTA.  In a
// warp, lane t takes row t of each 32-row chunk for the logits (its whole K row
// against the scaled queries, broadcast from shared memory), the chunk's
// weights then go round by shuffles for the value sum, where lane t owns
// d/32 dimensions (so the V rows are read coalesced).  Online softmax in base 2
// per head; the four warps, then the row splits, are merged with the usual
// rescaling.  Each warp's 32 value rows are copied into shared memory
// (cp.async) while the lanes compute the chunk's logits, so the value sum
// reads no global memory.  HBM-bound: every retained K and V row is read once.
#include "common.cuh"
#include "launch.h"

namespace tgvkv {
namespace {

constexpr int kDecThreads = 128;
constexpr int kDecWarps = kDecThreads / 32;

__device__ __forceinline__ float bf16_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }

// STAGE: value rows staged through shared memory (GQA: several heads share a
// row, so the row loop is long enough for the copies to pay); else read
// straight from global memory (one head per KV head: occupancy hides them).
template <int D, int GB, bool STAGE>
__global__ void __launch_bounds__(kDecThreads)
decode_kernel(Problem p, const uint16_t* __restrict__ q, const uint4* __restrict__ k_rows,
              const uint16_t* __restrict__ v_rows, const int64_t* __restrict__ offsets, int splits,
              float* __restrict__ out, float* __restrict__ part) {
    constexpr int DPL = D / 32;                 // value dims per lane (2 or 4)
    __shared__ __align__(16) float qs[GB][D];   // scaled queries of the CTA's heads
    __shared__ float wm[kDecWarps][GB], wl[kDecWarps][GB];
    // each warp's chunk of 32 value rows, copied in while its logits are computed;
    // after the row loop the same bytes hold the warps' partial sums
    constexpr size_t kVbuf = STAGE ? sizeof(uint16_t) * kDecWarps * 32 * D : 16;
    constexpr size_t kWacc = sizeof(float) * kDecWarps * GB * D;
    __shared__ __align__(16) unsigned char sbuf[kVbuf > kWacc ? kVbuf : kWacc];
    auto vbuf = reinterpret_cast<uint16_t (*)[32][D]>(sbuf);
    auto wacc = reinterpret_cast<float (*)[GB][D]>(sbuf);

    const int lg = blockIdx.x, split = blockIdx.y, hb = blockIdx.z;
    const int l = lg / p.H_kv, g = lg % p.H_kv;
    const int h0 = g * p.G + hb * GB;                     // first query head of this CTA
    const int nh = min(GB, p.G - hb * GB);                // heads of this CTA
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    for (int i = tid; i < GB * D; i += kDecThreads) {
        const int hh = i / D, c = i % D;
        float x = 0.f;
        if (hh < nh) {
            const uint16_t b = q[((size_t)l * p.H_q + h0 + hh) * D + c];
            x = __uint_as_float((uint32_t)b << 16) * p.scale_log2;
        }
        qs[hh][c] = x;
    }
    const long long lo = offsets[lg], hi = offsets[lg + 1];
    const long long len = hi > lo ? hi - lo : 0;
    const long long chunk = (len + splits - 1) / splits;
    const long long r0 = lo + (long long)split * chunk;
    const long long r1 = min(hi, r0 + chunk);
    __syncthreads();

    float m[GB], lsum[GB], acc[GB][DPL];
#pragma unroll
    for (int i = 0; i < GB; ++i) {
        m[i] = -INFINITY;
        lsum[i] = 0.f;
#pragma unroll
        for (int c = 0; c < DPL; ++c) acc[i][c] = 0.f;
    }
    for (long long base = r0 + (long long)warp * 32; base < r1; base += kDecWarps * 32) {
        const long long r = base + lane;
        const bool valid = r < r1;
        const int nrows = (int)min((long long)32, r1 - base);
        // value rows of the chunk into shared memory (16-byte copies, no wait yet)
        if (STAGE) {
            constexpr int PIECES = D / 8;                 // 16-byte pieces per row
            const char* src0 = reinterpret_cast<const char*>(v_rows) + (size_t)base * D * 2;
#pragma unroll
            for (int i = 0; i < PIECES; ++i) {
                const int piece = lane + 32 * i, row = piece / PIECES, col = piece % PIECES;
                if (row < nrows) {
                    const uint32_t dst = static_cast<uint32_t>(
                        __cvta_generic_to_shared(&vbuf[warp][row][col * 8]));
                    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst),
                                 "l"(src0 + (size_t)row * D * 2 + col * 16)
                                 : "memory");
                }
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
        }
        // logits of this lane's row for every head of the CTA
        float s[GB];
#pragma unroll
        for (int i = 0; i < GB; ++i) s[i] = 0.f;
        if (valid) {
            const uint4* kr = k_rows + (size_t)r * (D / 8);
#pragma unroll 4
            for (int c8 = 0; c8 < D / 8; ++c8) {
                const uint4 kv = __ldg(kr + c8);
                const float k0 = bf16_lo(kv.x), k1 = bf16_hi(kv.x), k2 = bf16_lo(kv.y), k3 = bf16_hi(kv.y);
                const float k4 = bf16_lo(kv.z), k5 = bf16_hi(kv.z), k6 = bf16_lo(kv.w), k7 = bf16_hi(kv.w);
#pragma unroll
                for (int i = 0; i < GB; ++i) {
                    const float4 qa = *reinterpret_cast<const float4*>(&qs[i][8 * c8]);
                    const float4 qb = *reinterpret_cast<const float4*>(&qs[i][8 * c8 + 4]);
                    s[i] = fmaf(k0, qa.x, fmaf(k1, qa.y, fmaf(k2, qa.z, fmaf(k3, qa.w, s[i]))));
                    s[i] = fmaf(k4, qb.x, fmaf(k5, qb.y, fmaf(k6, qb.z, fmaf(k7, qb.w, s[i]))));
                }
            }
        }
        float pr[GB];
#pragma unroll
        for (int i = 0; i < GB; ++i) {
            float cm = valid ? s[i] : -INFINITY;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) cm = fmaxf(cm, __shfl_xor_sync(~0u, cm, o));
            const float mn = fmaxf(m[i], cm);
            const float a = fast_exp2(m[i] - mn);      // 0 on the first chunk (m = -inf)
            pr[i] = valid ? fast_exp2(s[i] - mn) : 0.f;
            lsum[i] = lsum[i] * a + pr[i];
#pragma unroll
            for (int c = 0; c < DPL; ++c) acc[i][c] *= a;
            m[i] = mn;
        }
        if (STAGE) {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
            __syncwarp();
        }
        // value sum: the chunk's rows in turn, lane t owning dims DPL*t .. (unrolled
        // so that several rows' loads are in flight)
#pragma unroll 4
        for (int t = 0; t < nrows; ++t) {
            float vf[DPL];
            if (!STAGE) {
                const uint2 vv = __ldg(reinterpret_cast<const uint2*>(v_rows) +
                                       (size_t)(base + t) * (D / 4) + (DPL == 4 ? lane : lane / 2));
                if (DPL == 4) {
                    vf[0] = bf16_lo(vv.x);
                    vf[1] = bf16_hi(vv.x);
                    vf[2 % DPL] = bf16_lo(vv.y);
                    vf[3 % DPL] = bf16_hi(vv.y);
                } else {
                    const uint32_t w = (lane & 1) ? vv.y : vv.x;
                    vf[0] = bf16_lo(w);
                    vf[1 % DPL] = bf16_hi(w);
                }
            } else if (DPL == 4) {
                const uint2 vv = *reinterpret_cast<const uint2*>(&vbuf[warp][t][4 * lane]);
                vf[0] = bf16_lo(vv.x);
                vf[1] = bf16_hi(vv.x);
                vf[2 % DPL] = bf16_lo(vv.y);
                vf[3 % DPL] = bf16_hi(vv.y);
            } else {
                const uint32_t w = *reinterpret_cast<const uint32_t*>(&vbuf[warp][t][2 * lane]);
                vf[0] = bf16_lo(w);
                vf[1 % DPL] = bf16_hi(w);
            }
#pragma unroll
            for (int i = 0; i < GB; ++i) {
                const float pt = __shfl_sync(~0u, pr[i], t);
#pragma unroll
                for (int c = 0; c < DPL; ++c) acc[i][c] = fmaf(pt, vf[c], acc[i][c]);
            }
        }
        __syncwarp();   // every lane is done with vbuf before the next chunk's copies
    }
    // merge the four warps (sbuf changes role: every warp is done with its rows)
    __syncthreads();
#pragma unroll
    for (int i = 0; i < GB; ++i) {
        float ls = lsum[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ls += __shfl_xor_sync(~0u, ls, o);
        if (lane == 0) {
            wm[warp][i] = m[i];
            wl[warp][i] = ls;
        }
#pragma unroll
        for (int c = 0; c < DPL; ++c) wacc[warp][i][DPL * lane + c] = acc[i][c];
    }
    __syncthreads();
    for (int e = tid; e < GB * D; e += kDecThreads) {
        const int i = e / D, c = e % D;
        if (i >= nh) continue;
        float mt = -INFINITY;
        for (int w = 0; w < kDecWarps; ++w) mt = fmaxf(mt, wm[w][i]);
        float lt = 0.f, at = 0.f;
        if (mt != -INFINITY) {
            for (int w = 0; w < kDecWarps; ++w) {
                const float f = fast_exp2(wm[w][i] - mt);
                lt += wl[w][i] * f;
                at += wacc[w][i][c] * f;
            }
        }
        const int h = h0 + i;
        if (splits == 1) {
            out[((size_t)l * p.H_q + h) * D + c] = lt > 0.f ? at / lt : 0.f;
        } else {
            float* pp = part + (((size_t)l * p.H_q + h) * splits + split) * (D + 2);
            pp[c] = at;
            if (c == 0) {
                pp[D] = mt;
                pp[D + 1] = lt;
            }
        }
    }
}

// Merge the row splits of every (layer, query head).
template <int D>
__global__ void __launch_bounds__(D)
decode_merge_kernel(Problem p, int splits, const float* __restrict__ part, float* __restrict__ out) {
    const int lh = blockIdx.x, c = threadIdx.x;
    const float* pp = part + (size_t)lh * splits * (D + 2);
    float mt = -INFINITY;
    for (int s = 0; s < splits; ++s) mt = fmaxf(mt, pp[(size_t)s * (D + 2) + D]);
    float lt = 0.f, at = 0.f;
    if (mt != -INFINITY) {
        for (int s = 0; s < splits; ++s) {
            const float* q = pp + (size_t)s * (D + 2);
            const float f = fast_exp2(q[D] - mt);
            lt += q[D + 1] * f;
            at += q[c] * f;
        }
    }
    out[(size_t)lh * D + c] = lt > 0.f ? at / lt : 0.f;
}

template <int D, int GB>
cudaError_t launch_dec(const Problem& p, const uint16_t* q, const uint16_t* k_rows,
                       const uint16_t* v_rows, const int64_t* offsets, float* out, float* part,
                       cudaStream_t stream) {
    const int splits = decode_splits(p);
    const dim3 grid(p.L * p.H_kv, splits, (p.G + GB - 1) / GB);
    decode_kernel<D, GB, (GB > 1)><<<grid, kDecThreads, 0, stream>>>(
        p, q, reinterpret_cast<const uint4*>(k_rows), v_rows,
        offsets, splits, out, part);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || splits == 1) return e;
    decode_merge_kernel<D><<<p.L * p.H_q, D, 0, stream>>>(p, splits, part, out);
    return cudaGetLastError();
}

template <int D>
cudaError_t launch_dec_d(const Problem& p, const uint16_t* q, const uint16_t* k_rows,
                         const uint16_t* v_rows, const int64_t* offsets, float* out, float* part,
                         cudaStream_t stream) {
    if (p.G == 1) return launch_dec<D, 1>(p, q, k_rows, v_rows, offsets, out, part, stream);
    if (p.G == 2) return launch_dec<D, 2>(p, q, k_rows, v_rows, offsets, out, part, stream);
    if (p.G <= 4) return launch_dec<D, 4>(p, q, k_rows, v_rows, offsets, out, part, stream);
    return launch_dec<D, 8>(p, q, k_rows, v_rows, offsets, out, part, stream);
}

}  // namespace

cudaError_t launch_decode(const Problem& p, const uint16_t* q, const uint16_t* k_rows,
                          const uint16_t* v_rows, const int64_t* offsets, float* out, float* part,
                          cudaStream_t stream) {
    if (p.d == 64) return launch_dec_d<64>(p, q, k_rows, v_rows, offsets, out, part, stream);
    return launch_dec_d<128>(p, q, k_rows, v_rows, offsets, out, part, stream);
}

int decode_launches(const Problem& p) { return decode_splits(p) > 1 ? 2 : 1; }

}  // namespace tgvkv
