// Per-row softmax statistics over 32-key words of a TMEM accumulator row,
// shared by the score kernels: the online maximum m, normaliser Z and vision
// mass V of one query row (Eq. 2 rows, Eq. 5 / Eq. 6 vision slice), in base-2
// units (logits scaled by softmax_scale * log2 e).
#pragma once

#include <math.h>

#include "common.cuh"

namespace tgvkv {

__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

__device__ __forceinline__ float max32(const float (&x)[32]) {
    float a = fmax3(x[0], x[1], x[2]), b = fmax3(x[3], x[4], x[5]), c = fmax3(x[6], x[7], x[8]);
    float d = fmax3(x[9], x[10], x[11]), e = fmax3(x[12], x[13], x[14]);
    float f = fmax3(x[15], x[16], x[17]), g = fmax3(x[18], x[19], x[20]);
    float h = fmax3(x[21], x[22], x[23]), i = fmax3(x[24], x[25], x[26]);
    float j = fmax3(x[27], x[28], x[29]), k = fmaxf(x[30], x[31]);
    a = fmax3(a, b, c);
    d = fmax3(d, e, f);
    g = fmax3(g, h, i);
    j = fmaxf(j, k);
    return fmaxf(fmax3(a, d, g), j);
}

__device__ __forceinline__ float max32_masked(const float (&x)[32], int lim) {
    float a = -INFINITY, b = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
        if (i <= lim) a = fmaxf(a, x[i]);
        if (i + 1 <= lim) b = fmaxf(b, x[i + 1]);
    }
    return fmaxf(a, b);
}

// Sum of e_c = 2^(x_c sl2 + nm) over one 32-key word (columns c <= lim when
// MASKED), and the part of it over the vision keys flagged in vm.  Exponent
// arguments and sums run on packed fp32 pairs.
template <bool MASKED>
__device__ __forceinline__ void exp_word(const float (&x)[32], float sl2, float nm, int lim,
                                         uint32_t vm, float& z, float& v) {
    const float2 s2 = make_float2(sl2, sl2), n2 = make_float2(nm, nm);
    float2 za = make_float2(0.f, 0.f), zb = za;
    if (vm == 0u || vm == 0xFFFFFFFFu) {
#pragma unroll
        for (int c = 0; c < 32; c += 4) {
            const float2 t0 = fma2(make_float2(x[c], x[c + 1]), s2, n2);
            const float2 t1 = fma2(make_float2(x[c + 2], x[c + 3]), s2, n2);
            float2 e0 = make_float2(fast_exp2(t0.x), fast_exp2(t0.y));
            float2 e1 = make_float2(fast_exp2(t1.x), fast_exp2(t1.y));
            if (MASKED) {
                if (c > lim) e0.x = 0.f;
                if (c + 1 > lim) e0.y = 0.f;
                if (c + 2 > lim) e1.x = 0.f;
                if (c + 3 > lim) e1.y = 0.f;
            }
            za = add2(za, e0);
            zb = add2(zb, e1);
        }
        const float zs = (za.x + za.y) + (zb.x + zb.y);
        z += zs;
        if (vm) v += zs;
    } else {
        float2 va = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
            const float2 t = fma2(make_float2(x[c], x[c + 1]), s2, n2);
            float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
            if (MASKED) {
                if (c > lim) e.x = 0.f;
                if (c + 1 > lim) e.y = 0.f;
            }
            za = add2(za, e);
            va = add2(va, make_float2((vm >> c) & 1u ? e.x : 0.f, (vm >> (c + 1)) & 1u ? e.y : 0.f));
        }
        z += za.x + za.y;
        v += va.x + va.y;
    }
}

// exp_word plus the sum over the visible keys NOT in vm (u): the text-key pass
// keeps the vision mass of each row this way, for the vision pass to reuse.
template <bool MASKED>
__device__ __forceinline__ void exp_word_both(const float (&x)[32], float sl2, float nm, int lim,
                                              uint32_t vm, float& z, float& v, float& u) {
    if (vm == 0u || vm == 0xFFFFFFFFu) {
        float zs = 0.f;
        exp_word<MASKED>(x, sl2, nm, lim, 0u, zs, zs);   // (v untouched when vm == 0)
        z += zs;
        if (vm) v += zs;
        else u += zs;
    } else {
        const float2 s2 = make_float2(sl2, sl2), n2 = make_float2(nm, nm);
        float2 za = make_float2(0.f, 0.f), va = za, ua = za;
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
            const float2 t = fma2(make_float2(x[c], x[c + 1]), s2, n2);
            float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
            if (MASKED) {
                if (c > lim) e.x = 0.f;
                if (c + 1 > lim) e.y = 0.f;
            }
            za = add2(za, e);
            const bool b0 = (vm >> c) & 1u, b1 = (vm >> (c + 1)) & 1u;
            va = add2(va, make_float2(b0 ? e.x : 0.f, b1 ? e.y : 0.f));
            ua = add2(ua, make_float2(b0 ? 0.f : e.x, b1 ? 0.f : e.y));
        }
        z += za.x + za.y;
        v += va.x + va.y;
        u += ua.x + ua.y;
    }
}

// Online statistics of one row over one 32-key word: columns 0..lim visible.
// The row keeps a reference m (base-2 units) and sums its terms 2^(x sl2 - m):
// the row's first visible word sets m to that word's maximum; a later word
// keeps m unless its terms against m sum above kWordSumLimit (some term large,
// or overflowed), and is then taken again against its own maximum, which moves
// m up (z and v rescaled).  Any reference gives the same attention entries
// 2^(x sl2 - m) / Z; this one never exceeds the row's maximum and keeps every
// term at most kWordSumLimit, and most words skip the 32-key maximum.
constexpr float kWordSumLimit = 32.f * 256.f;

__device__ __forceinline__ void row_word(const float (&x)[32], float sl2, int lim, uint32_t vm,
                                         float& m, float& z, float& v) {
    if (lim < 0) return;
    if (m != -INFINITY) {
        float zs = 0.f, vs = 0.f;
        if (lim >= 31)
            exp_word<false>(x, sl2, -m, 31, vm, zs, vs);
        else
            exp_word<true>(x, sl2, -m, lim, vm, zs, vs);
        if (zs <= kWordSumLimit) {   // false for inf and nan too
            z += zs;
            v += vs;
            return;
        }
    }
    const float m_new = fmaxf(m, (lim >= 31 ? max32(x) : max32_masked(x, lim)) * sl2);
    const float alpha = fast_exp2(m - m_new);   // m = -inf: alpha = 0, z = v = 0 stay 0
    z *= alpha;
    v *= alpha;
    if (lim >= 31)
        exp_word<false>(x, sl2, -m_new, 31, vm, z, v);
    else
        exp_word<true>(x, sl2, -m_new, lim, vm, z, v);
    m = m_new;
}

// row_word with the complement mass u as well (text-key pass: the visible keys
// not in vm).
__device__ __forceinline__ void row_word_both(const float (&x)[32], float sl2, int lim, uint32_t vm,
                                              float& m, float& z, float& v, float& u) {
    if (lim < 0) return;
    if (m != -INFINITY) {
        float zs = 0.f, vs = 0.f, us = 0.f;
        if (lim >= 31)
            exp_word_both<false>(x, sl2, -m, 31, vm, zs, vs, us);
        else
            exp_word_both<true>(x, sl2, -m, lim, vm, zs, vs, us);
        if (zs <= kWordSumLimit) {
            z += zs;
            v += vs;
            u += us;
            return;
        }
    }
    const float m_new = fmaxf(m, (lim >= 31 ? max32(x) : max32_masked(x, lim)) * sl2);
    const float alpha = fast_exp2(m - m_new);
    z *= alpha;
    v *= alpha;
    u *= alpha;
    if (lim >= 31)
        exp_word_both<false>(x, sl2, -m_new, 31, vm, z, v, u);
    else
        exp_word_both<true>(x, sl2, -m_new, lim, vm, z, v, u);
    m = m_new;
}

}  // namespace tgvkv
