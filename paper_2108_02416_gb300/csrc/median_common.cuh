// Pieces of the coordinate-wise aggregation (aggregate.cu): the totalOrder
// key map, the value-space bin map, tag matching, compensated sums and the
// search modes of the lower median.
#pragma once

#include <stdint.h>

namespace aspis {

constexpr int kNB = 128;          // key-space histogram rows of the exact path
constexpr int kLogNB = 7;         // key bits resolved per key-space pass
constexpr int kVB = 256;          // value-space histogram rows
constexpr int kTopBin = 254;      // value-space bins are 0..kTopBin
constexpr uint32_t kPadTag = 0xFFu;   // tag byte of a missing row: no value-space bin

// IEEE totalOrder as unsigned order: flip all bits of negatives, the sign
// bit of non-negatives.  A bijection, so the median's bits come back exactly.
__device__ __forceinline__ uint32_t to_key(uint32_t u)
{
    return u ^ ((uint32_t)((int32_t)u >> 31) | 0x80000000u);
}

__device__ __forceinline__ uint32_t from_key(uint32_t k)
{
    return k ^ ((uint32_t)((int32_t)~k >> 31) | 0x80000000u);
}

// Value-space bin of x, as the bits of 2^23 + bin: y = sat(x*s + c) in
// [0, 1] (fma with saturation: NaN gives +0), then 2^23 + rint(254*y), whose
// low byte is the bin 0..254.  Both steps are correctly rounded and
// non-decreasing, so the map is monotone in the IEEE totalOrder of every
// non-NaN x (+0 and -0 share a bin) and always lands in 0..126, whatever s
// and c are.  NaNs are detected separately.
__device__ __forceinline__ uint32_t vbin_bits(float x, float s, float c)
{
    float y;
    asm("fma.rn.sat.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(x), "f"(s), "f"(c));
    return __float_as_uint(fmaf(y, (float)kTopBin, 8388608.0f));
}

enum { M_DONE = 0, M_VH, M_VC, M_VM, M_KA, M_KH, M_KC };

// Four tag bytes against the target bytes of vbx: 0x80 in each byte whose tag
// equals its target, 0 elsewhere.  Exact for every byte value: the sum of a
// byte's low seven bits and 0x7F sets its top bit iff they are not all zero
// and cannot carry into the next byte.  (Targets of coordinates that search
// nothing are 0xFF, equal to the padding tag; callers skip such hits.)
__device__ __forceinline__ uint32_t tag_match(uint32_t w, uint32_t vbx)
{
    const uint32_t x = w ^ vbx;
    return ~(((x & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | x) & 0x80808080u;
}

// Two-sum: s + e == a + b exactly (Knuth); no products, so nothing to fuse.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e)
{
    s = a + b;
    const float bp = s - a;
    e = (a - (s - bp)) + (b - bp);
}

}  // namespace aspis
