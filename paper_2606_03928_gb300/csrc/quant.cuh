// Per-token asymmetric b-bit quantization of one value row (the equation of Sec. 4.4), one warp per row.
#pragma once

#include <cstdint>

namespace vase {

// Lane l holds dims 4l .. 4l+3 of a bf16 value row (one uint2).  The warp takes z = min v and
// s = (max v - min v) / (2^b - 1), then Q = round((v - z) / s), half to even, clamped to 0 .. 2^b - 1; the
// subtraction, the divisions and the rounding are each in fp32 (IEEE), and a row of equal values (s = 0) gets
// codes 0.  Lane l packs its four codes into 4b bits (dim 4l + e at bits e*b) at byte l*b/2 of the code row;
// lane 0 writes (s, z).  Every lane of the warp must call it.
__device__ __forceinline__ void quantize_row_warp(uint2 raw, int bits, int lane, uint8_t* code_row, float* sz) {
    const float v[4] = {__uint_as_float(raw.x << 16), __uint_as_float(raw.x & 0xFFFF0000u),
                        __uint_as_float(raw.y << 16), __uint_as_float(raw.y & 0xFFFF0000u)};
    float lo = fminf(fminf(v[0], v[1]), fminf(v[2], v[3]));
    float hi = fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3]));
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    const float levels = static_cast<float>((1 << bits) - 1);
    const float s = __fdiv_rn(__fsub_rn(hi, lo), levels);
    uint32_t packed = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float t = s > 0.f ? rintf(__fdiv_rn(__fsub_rn(v[e], lo), s)) : 0.f;
        const uint32_t c = static_cast<uint32_t>(fminf(fmaxf(t, 0.f), levels));
        packed |= c << (e * bits);
    }
    const int code_bytes = bits / 2;  // bytes of one lane's four codes
    uint8_t* dst = code_row + lane * code_bytes;
    if (code_bytes == 4) *reinterpret_cast<uint32_t*>(dst) = packed;
    else if (code_bytes == 2) *reinterpret_cast<uint16_t*>(dst) = static_cast<uint16_t>(packed);
    else *dst = static_cast<uint8_t>(packed);
    if (lane == 0) {
        sz[0] = s;
        sz[1] = lo;
    }
}

}  // namespace vase
