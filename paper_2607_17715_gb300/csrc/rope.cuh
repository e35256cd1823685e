// RoPE angles and the 2x2 rotation shared by the streaming kernels.  Channel i pairs with
// i + d/2 and turns by pos * theta^(-2i/d); the angle comes from the phase accumulator in
// RopeTurns (the low 64 bits of pos * turn[i] are the exact fractional turn) and sincospif.
#pragma once

#include <cstdint>

namespace c2kv {
namespace {

__device__ __forceinline__ float2 turn_cs(uint64_t turn, int64_t pos) {
    const uint64_t frac = (uint64_t)pos * turn;                 // turns mod 1, exact
    const float x = (float)(long long)frac * 0x1p-63f;          // 2 * turns in [-1, 1)
    float s, c;
    sincospif(x, &s, &c);
    return make_float2(c, s);
}

// (x, y) turned by the angle whose (cos, sin) is cs, with the rounding spelled out (one
// product rounded, then a fused multiply-add) so that every kernel that turns a pair gets
// the same bits.
__device__ __forceinline__ void rotate1(float x, float y, float2 cs, float& ox, float& oy) {
    ox = __fmaf_rn(x, cs.x, -__fmul_rn(y, cs.y));
    oy = __fmaf_rn(x, cs.y, __fmul_rn(y, cs.x));
}

template <int E>
__device__ __forceinline__ void rotate(const float* x, const float* y, const float2* cs,
                                       float* ox, float* oy) {
#pragma unroll
    for (int e = 0; e < E; ++e) rotate1(x[e], y[e], cs[e], ox[e], oy[e]);
}

}  // namespace
}  // namespace c2kv
