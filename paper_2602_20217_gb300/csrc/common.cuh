// Device helpers shared by the kernels of libknapspec (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#define KS_DEV __device__ __forceinline__

namespace ks {

constexpr int kWarp = 32;

// 16-byte streaming load that bypasses L1 (weights are read exactly once per pass).
KS_DEV uint4 ldg_stream(const void* p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

KS_DEV uint4 lds128(const void* p) {
    return *reinterpret_cast<const uint4*>(p);
}

// D = A * B + D, m16n8k16, bf16 inputs, fp32 accumulators.
// A (16x16, row-major) fragment a0..a3, B (16x8, column-major) fragment b0..b1.
KS_DEV void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                     uint32_t b0, uint32_t b1) {
    asm(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, "
        "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

KS_DEV float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
KS_DEV float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// Round two floats to bf16 (nearest even) and pack (lo in the low half).
KS_DEV uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

KS_DEV float to_float(float v) { return v; }
KS_DEV float to_float(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T> KS_DEV T from_float(float v);
template <> KS_DEV float from_float<float>(float v) { return v; }
template <> KS_DEV __nv_bfloat16 from_float<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

KS_DEV float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

KS_DEV float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Block-wide sum in a fixed order: per-warp butterfly, then warp 0 sums the
// warp totals in warp order.  Every thread gets the result.
template <int NWARPS>
KS_DEV float block_sum(float v, float* scratch /* >= NWARPS + 1 floats */) {
    v = warp_sum(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) scratch[w] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < NWARPS; ++i) s += scratch[i];
        scratch[NWARPS] = s;
    }
    __syncthreads();
    return scratch[NWARPS];
}

// (value, index) argmax merge: larger value wins, ties go to the smaller index.
KS_DEV bool better(float v, int i, float bv, int bi) {
    return v > bv || (v == bv && i < bi);
}

KS_DEV float silu(float z) { return z / (1.f + __expf(-z)); }

}  // namespace ks
