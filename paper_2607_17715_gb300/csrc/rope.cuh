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

template <int E>
__device__ __forceinline__ void rotate(const float* x, const float* y, const float2* cs,
                                       float* ox, float* oy) {
#pragma unroll
    for (int e = 0; e < E; ++e) {
        ox[e] = x[e] * cs[e].x - y[e] * cs[e].y;
        oy[e] = x[e] * cs[e].y + y[e] * cs[e].x;
    }
}

}  // namespace
}  // namespace c2kv
