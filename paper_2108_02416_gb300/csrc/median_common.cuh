// Pieces of the lower-median search (aggregate.cu): the totalOrder key map,
// the value-space bin map, tag matching and the search modes.
#pragma once

#include <stdint.h>

namespace aspis {

constexpr int kNB = 128;          // histogram bins per pass
constexpr int kLogNB = 7;
constexpr int kCap = 32;          // keys ranked directly

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

// Value-space bin of y = fma(x, s, c): the integer part of y read from its
// bits (y is near 2^23, where one unit is one ulp), clamped to [0, kNB).
// The clamp is done on the float (an integer offset of a negative y's bits
// would wrap), so negative y, -inf and underflow go to bin 0 and +inf or
// large y to kNB-1.  Rounding is monotone, so the map is monotone in the IEEE
// totalOrder of x for every non-NaN x.  NaNs are detected separately: fma
// returns a canonical NaN whatever the sign of x (and it lands in bin 0).
__device__ __forceinline__ uint32_t vbin(float y)
{
    const float yc = fminf(fmaxf(y, 8388608.0f), 8388608.0f + (float)(kNB - 1));
    return __float_as_uint(yc) - 0x4B000000u;
}

enum { M_DONE = 0, M_VH, M_VC, M_VM, M_VR, M_KA, M_KH, M_KC };

// Four tag bytes against the replicated bin vbx: 0x80 in each byte whose tag
// equals the bin.  Tags are < 0x80 and padding is 0xFF, so after the XOR a
// byte is zero exactly at a match; OR-ing 0x80 first keeps the per-byte
// subtraction from borrowing across bytes.
__device__ __forceinline__ uint32_t tag_match(uint32_t word, uint32_t vbx)
{
    const uint32_t x = word ^ vbx;
    return ~((x | 0x80808080u) - 0x01010101u) & ~x & 0x80808080u;
}

// Two-sum: s + e == a + b exactly (Knuth); no products, so nothing to fuse.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e)
{
    s = a + b;
    const float bp = s - a;
    e = (a - (s - bp)) + (b - bp);
}

}  // namespace aspis
