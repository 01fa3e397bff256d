// Device helpers shared by the kernel translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "sn_internal.h"

namespace sn {
namespace k {

template <typename T> __device__ __forceinline__ float ldf(const T *p);
template <> __device__ __forceinline__ float ldf<float>(const float *p) { return *p; }
template <> __device__ __forceinline__ float ldf<__half>(const __half *p) { return __half2float(*p); }
template <> __device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16 *p) {
    return __bfloat162float(*p);
}

// round-to-nearest-even stores
template <typename T> __device__ __forceinline__ void stf(T *p, float v);
template <> __device__ __forceinline__ void stf<float>(float *p, float v) { *p = v; }
template <> __device__ __forceinline__ void stf<__half>(__half *p, float v) { *p = __float2half_rn(v); }
template <> __device__ __forceinline__ void stf<__nv_bfloat16>(__nv_bfloat16 *p, float v) {
    *p = __float2bfloat16_rn(v);
}

template <typename T> __device__ __forceinline__ T cvt(float v);
template <> __device__ __forceinline__ float cvt<float>(float v) { return v; }
template <> __device__ __forceinline__ __half cvt<__half>(float v) { return __float2half_rn(v); }
template <> __device__ __forceinline__ __nv_bfloat16 cvt<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

// The common activations first, as before the hard-swish pair was added: in
// an unrolled epilogue every extra test of `act` is paid per element.
__device__ __forceinline__ float act_apply(float v, int act) {
    if (act == SN_ACT_RELU) return fmaxf(v, 0.0f);
    if (act == SN_ACT_NONE) return v;
    if (act == SN_ACT_RELU6) return fminf(fmaxf(v, 0.0f), 6.0f);
    const float t = fminf(fmaxf(v + 3.0f, 0.0f), 6.0f) / 6.0f;  // hard sigmoid
    return act == SN_ACT_HSWISH ? v * t : t;
}

// streaming multiprocessors of the current device (host)
inline int num_sms() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    }
    return n;
}

inline unsigned grid_for(int64_t n, int block, int64_t cap = 152LL * 64) {
    int64_t g = (n + block - 1) / block;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (unsigned)g;
}

// dispatch a runtime dtype to a C++ type
// Programmatic dependent launch.  Every kernel of the library is launched
// with launch_pdl, which lets it start (set up, fetch descriptors) while the
// previous kernel on the stream drains; the kernel calls griddep_wait()
// before its first global-memory access, which returns once the previous
// grid has completed and its writes are visible, and griddep_launch() to let
// its own successor start early.  Both are no-ops for a plain launch.
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

// acc += x * w on the two 16-bit lanes of x2 and w2, accumulating in f32 with
// the sm_100 mixed-precision FMA (fp32 destination, f16/bf16 factors).  The
// product of two f16 or two bf16 values is exact in f32, so each lane equals
// fmaf(float(x), float(w), acc) bit for bit, without the two conversions.
template <typename T>
__device__ __forceinline__ void mac2(float &a0, float &a1, uint32_t x2, uint32_t w2);
template <>
__device__ __forceinline__ void mac2<__half>(float &a0, float &a1, uint32_t x2, uint32_t w2) {
    asm("{\n\t.reg .b16 xl, xh, wl, wh;\n\tmov.b32 {xl, xh}, %2;\n\tmov.b32 {wl, wh}, %3;\n\t"
        "fma.rn.f32.f16 %0, xl, wl, %0;\n\tfma.rn.f32.f16 %1, xh, wh, %1;\n\t}"
        : "+f"(a0), "+f"(a1)
        : "r"(x2), "r"(w2));
}
template <>
__device__ __forceinline__ void mac2<__nv_bfloat16>(float &a0, float &a1, uint32_t x2, uint32_t w2) {
    asm("{\n\t.reg .b16 xl, xh, wl, wh;\n\tmov.b32 {xl, xh}, %2;\n\tmov.b32 {wl, wh}, %3;\n\t"
        "fma.rn.f32.bf16 %0, xl, wl, %0;\n\tfma.rn.f32.bf16 %1, xh, wh, %1;\n\t}"
        : "+f"(a0), "+f"(a1)
        : "r"(x2), "r"(w2));
}

// Division by a divisor fixed at launch, for numerators below 2^31:
// q = (umulhi(n, m) + n) >> l with l = ceil(log2 d), m = floor(2^32 (2^l - d) / d) + 1
// (the round-up multiplier method of Granlund and Montgomery).  The generic
// 32-bit division is a dependent chain of ~20 instructions, 64-bit division a
// library call.
struct FastDiv {
    uint32_t d, m, l;
};
inline FastDiv make_fastdiv(uint32_t d) {
    uint32_t l = 0;
    while ((1ull << l) < d) ++l;
    const uint64_t m = ((1ull << 32) * ((1ull << l) - d)) / d + 1;
    return FastDiv{d, (uint32_t)m, l};
}
__device__ __forceinline__ uint32_t fdiv(uint32_t n, const FastDiv &f) {
    return (uint32_t)(((uint64_t)__umulhi(n, f.m) + n) >> f.l);
}

#define SN_DT_SWITCH(dt, T, ...)                          \
    switch (dt) {                                         \
    case SN_F32: { using T = float; __VA_ARGS__; break; } \
    case SN_F16: { using T = __half; __VA_ARGS__; break; } \
    default: { using T = __nv_bfloat16; __VA_ARGS__; break; } \
    }

struct ConvDims {
    int32_t N, C, H, W, K, P, Q, R, S, sh, sw, ph, pw, dh, dw, groups, act;
};

// NHWC 3x3 depthwise through a TMA-fed shared-memory ring of input rows
bool dw3_ring_applies(const LaunchArgs &a, const ConvDims &d);
cudaError_t dw3_nhwc_ring(const LaunchArgs &a, const ConvDims &d);

cudaError_t conv_wino_buffers(const ConvDims &d, sn_schema s, const void *x, const void *u, const float *bias,
                              void *y, float *V, float *Mx, cudaStream_t st);

inline ConvDims conv_dims(const LaunchArgs &a) {
    const sn_conv_params &p = a.layer->conv;
    const Shape &i = a.in_shapes[0];
    const Shape &o = a.layer->out;
    return ConvDims{(int32_t)i.n, (int32_t)i.c, (int32_t)i.h, (int32_t)i.w, (int32_t)o.c, (int32_t)o.h,
                    (int32_t)o.w, p.kh, p.kw, p.sh, p.sw, p.ph, p.pw, p.dh, p.dw, p.groups, p.act};
}

}  // namespace k
}  // namespace sn
