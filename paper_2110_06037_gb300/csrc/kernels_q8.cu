// Routines and adapts of the qint8 schema (section II-C quantisation; the
// hybrid float/qint8 tuning of section V-C).
//
// A qint8 blob holds int8 codes q with one scale s > 0 per blob (symmetric,
// offset 0): it stands for the values q * s.  Weights carry one scale per
// output channel, s_w[k] = max |W[k, .]| / 127.  A routine sums code
// products exactly in int32 and requantises in fp32, one rounding per written
// operation (no fused multiply-add, __f*_rn throughout):
//     y = float(acc) * (s_x * s_w[k]) + bias[k]  [+ q_r * s_r]
//     q_y = clamp(rint(act(y) * (1 / s_y)), -127, 127)
// so that the codes are a deterministic function of the inputs.
//
// Integer dot products use dp4a (four int8 products added into an int32 per
// instruction) on the CUDA cores.
#include <cmath>
#include <type_traits>

#include "kern_common.cuh"

namespace sn {
namespace k {

namespace {

constexpr int QMAX = 127;

__device__ __forceinline__ int8_t q8_code(float y, float inv) {
    const int q = __float2int_rn(__fmul_rn(y, inv));
    return (int8_t)max(-QMAX, min(QMAX, q));
}

// the fused activations with one rounding per operation
__device__ __forceinline__ float q8_act(float v, int act) {
    if (act == SN_ACT_RELU) return fmaxf(v, 0.0f);
    if (act == SN_ACT_NONE) return v;
    if (act == SN_ACT_RELU6) return fminf(fmaxf(v, 0.0f), 6.0f);
    const float t = __fdiv_rn(fminf(fmaxf(__fadd_rn(v, 3.0f), 0.0f), 6.0f), 6.0f);  // hard sigmoid
    return act == SN_ACT_HSWISH ? __fmul_rn(v, t) : t;
}

// act(float(acc) * (s_x * s_w) + bias [+ residual value]) in fp32
__device__ __forceinline__ float q8_value(int acc, float s_x, float s_w, float bias, float resid, int act) {
    float y = __fadd_rn(__fmul_rn(__int2float_rn(acc), __fmul_rn(s_x, s_w)), bias);
    y = __fadd_rn(y, resid);
    return q8_act(y, act);
}

// the output element: a code of the output blob's scale, or, when the routine
// writes a float schema (dequantisation fused into the epilogue), the fp32
// value rounded to that type
template <typename TO>
__device__ __forceinline__ TO q8_out(float y, float inv) {
    if constexpr (std::is_same<TO, int8_t>::value) return q8_code(y, inv);
    else return cvt<TO>(y);
}

__device__ __forceinline__ int dp4a(int a, int b, int c) { return __dp4a(a, b, c); }

inline size_t align16(int64_t n) { return (size_t)((n + 15) / 16 * 16); }

// per-output-channel weight scales follow the codes, 16-byte aligned
inline const float *wscales(const void *wt, int64_t elems) {
    return reinterpret_cast<const float *>(static_cast<const char *>(wt) + align16(elems));
}

}  // namespace

size_t q8_weight_bytes(int64_t K, int64_t elems) { return align16(elems) + (size_t)K * sizeof(float); }

// ===========================================================================
// adapts: quantise, dequantise, layout permutation of codes
// ===========================================================================
// element transform of a conversion: codes stay codes, a float value becomes
// a code of scale s, a code becomes its value q * s
template <typename Ti, typename To>
__device__ __forceinline__ To q8_xform(Ti v, float s, float inv) {
    if constexpr (std::is_same<Ti, int8_t>::value && std::is_same<To, int8_t>::value) {
        return v;
    } else if constexpr (std::is_same<Ti, int8_t>::value) {
        return cvt<To>(__fmul_rn((float)v, s));
    } else {
        static_assert(std::is_same<To, int8_t>::value, "one side of a qint8 adapt is qint8");
        return q8_code(ldf<Ti>(&v), inv);
    }
}

template <typename Ti, typename To>
__global__ void q8_cast_kernel(const Ti *__restrict__ x, To *__restrict__ y, int64_t n, float s, float inv) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        y[i] = q8_xform<Ti, To>(x[i], s, inv);
}

// four consecutive elements per thread (n % 4 == 0; bases aligned to 4
// elements of each side)
template <typename T, int N> struct alignas(sizeof(T) * N) Vec { T v[N]; };

template <typename Ti, typename To>
__global__ void q8_cast4_kernel(const Vec<Ti, 4> *__restrict__ x, Vec<To, 4> *__restrict__ y, int64_t n4, float s,
                                float inv) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const Vec<Ti, 4> a = x[i];
        Vec<To, 4> b;
#pragma unroll
        for (int e = 0; e < 4; ++e) b.v[e] = q8_xform<Ti, To>(a.v[e], s, inv);
        y[i] = b;
    }
}

// the value a conversion stores, as a float: a code (exact) when the output is
// qint8, the fp32 value q * s when the input is
template <typename Ti, typename To>
__device__ __forceinline__ float q8_pre(float v, float s, float inv) {
    if constexpr (std::is_same<Ti, int8_t>::value && std::is_same<To, int8_t>::value) return v;
    else if constexpr (std::is_same<Ti, int8_t>::value) return __fmul_rn(v, s);
    else return (float)q8_code(v, inv);
}

template <typename T> __device__ __forceinline__ float q8_ld(const T *p) { return ldf<T>(p); }
template <> __device__ __forceinline__ float q8_ld<int8_t>(const int8_t *p) { return (float)*p; }
template <typename T> __device__ __forceinline__ T q8_cv(float v) { return cvt<T>(v); }
template <> __device__ __forceinline__ int8_t q8_cv<int8_t>(float v) { return (int8_t)(int)v; }

template <typename T, int VB>
struct QVec {
    static constexpr int E = VB / (int)sizeof(T);
    using V = typename std::conditional<
        VB == 16, uint4,
        typename std::conditional<VB == 8, uint2,
                                  typename std::conditional<VB == 4, uint32_t,
                                                            typename std::conditional<VB == 2, uint16_t,
                                                                                      uint8_t>::type>::type>::type>::type;
    __device__ __forceinline__ static void load(const T *p, float (&f)[E]) {
        const V v = *reinterpret_cast<const V *>(p);
        const T *t = reinterpret_cast<const T *>(&v);
#pragma unroll
        for (int e = 0; e < E; ++e) f[e] = q8_ld<T>(t + e);
    }
    __device__ __forceinline__ static void store(T *p, const float (&f)[E]) {
        V v;
        T *t = reinterpret_cast<T *>(&v);
#pragma unroll
        for (int e = 0; e < E; ++e) t[e] = q8_cv<T>(f[e]);
        *reinterpret_cast<V *>(p) = v;
    }
};

// same layout, 16 elements per thread (n % 16 == 0, 16-byte aligned bases)
template <typename Ti, typename To>
__global__ void q8_cast16_kernel(const Ti *__restrict__ x, To *__restrict__ y, int64_t n16, float s, float inv) {
    griddep_launch();
    griddep_wait();
    constexpr int EI = 16 / (int)sizeof(Ti), EO = 16 / (int)sizeof(To);
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16;
         i += (int64_t)gridDim.x * blockDim.x) {
        float f[16];
#pragma unroll
        for (int k = 0; k < 16 / EI; ++k) {
            float g[EI];
            QVec<Ti, 16>::load(x + i * 16 + k * EI, g);
#pragma unroll
            for (int e = 0; e < EI; ++e) f[k * EI + e] = q8_pre<Ti, To>(g[e], s, inv);
        }
#pragma unroll
        for (int k = 0; k < 16 / EO; ++k) {
            float g[EO];
#pragma unroll
            for (int e = 0; e < EO; ++e) g[e] = f[k * EO + e];
            QVec<To, 16>::store(y + i * 16 + k * EO, g);
        }
    }
}

// y[b][c][r] = f(x[b][r][c]) through a 64 x 64 shared-memory tile, VBI-byte
// vectors along the input rows and VBO-byte vectors along the output rows
constexpr int QT = 64;
template <typename Ti, typename To, int VBI, int VBO>
__global__ void __launch_bounds__(256) q8_transpose_vec_kernel(const Ti *__restrict__ x, To *__restrict__ y,
                                                               int64_t R, int64_t Cc, float s, float inv) {
    griddep_launch();
    griddep_wait();
    using LI = QVec<Ti, VBI>;
    using LO = QVec<To, VBO>;
    constexpr int EI = LI::E, EO = LO::E;
    __shared__ float tile[QT][QT + 1];
    const int64_t b = blockIdx.z;
    const int64_t r0 = (int64_t)blockIdx.y * QT, c0 = (int64_t)blockIdx.x * QT;
    const Ti *xb = x + b * R * Cc;
    To *yb = y + b * R * Cc;
    constexpr int VI = QT / EI;
#pragma unroll 4
    for (int i = threadIdx.x; i < QT * VI; i += 256) {
        const int row = i / VI, cv = i % VI;
        const int64_t r = r0 + row, c = c0 + cv * EI;
        if (r < R && c < Cc) {
            float f[EI];
            LI::load(xb + r * Cc + c, f);
#pragma unroll
            for (int e = 0; e < EI; ++e) tile[row][cv * EI + e] = q8_pre<Ti, To>(f[e], s, inv);
        }
    }
    __syncthreads();
    constexpr int VO = QT / EO;
#pragma unroll 4
    for (int i = threadIdx.x; i < QT * VO; i += 256) {
        const int orow = i / VO, ov = i % VO;
        const int64_t c = c0 + orow, r = r0 + ov * EO;
        if (c < Cc && r < R) {
            float f[EO];
#pragma unroll
            for (int e = 0; e < EO; ++e) f[e] = tile[ov * EO + e][orow];
            LO::store(yb + c * R + r, f);
        }
    }
}

// widest vector (16, 8 or 4 bytes, else one element) that every row of n
// elements of es bytes from an aligned base admits, and at most 64 elements
static int q8_row_vec(int64_t n, int es, const void *base) {
    for (int vb : {16, 8, 4})
        if (vb / es <= QT && vb >= es && (n * es) % vb == 0 && (uintptr_t)base % vb == 0) return vb;
    return es;
}

template <typename Ti, typename To, int VBI>
static void launch_q8_transpose(int vo, dim3 grid, cudaStream_t st, const Ti *x, To *y, int64_t R, int64_t Cc,
                                float s, float inv) {
    constexpr int SO = (int)sizeof(To);
    if (vo == 16) launch_pdl(q8_transpose_vec_kernel<Ti, To, VBI, 16>, grid, 256, 0, st, x, y, R, Cc, s, inv);
    else if (vo == 8) launch_pdl(q8_transpose_vec_kernel<Ti, To, VBI, 8>, grid, 256, 0, st, x, y, R, Cc, s, inv);
    else if (vo == 4) launch_pdl(q8_transpose_vec_kernel<Ti, To, VBI, (SO <= 4 ? 4 : SO)>, grid, 256, 0, st, x, y, R,
                                 Cc, s, inv);
    else launch_pdl(q8_transpose_vec_kernel<Ti, To, VBI, SO>, grid, 256, 0, st, x, y, R, Cc, s, inv);
}

template <typename Ti, typename To>
static cudaError_t convert_q8_t(const void *x, int lay_in, void *y, int lay_out, Shape sh, float s, float inv,
                                cudaStream_t st) {
    const int64_t n = sh.numel();
    if (n == 0) return cudaSuccess;
    if (lay_in == lay_out || sh.c == 1 || sh.h * sh.w == 1) {
        if (n % 16 == 0 && (uintptr_t)x % 16 == 0 && (uintptr_t)y % 16 == 0) {
            launch_pdl(q8_cast16_kernel<Ti, To>, grid_for(n / 16, 256), 256, 0, st, (const Ti *)x, (To *)y, n / 16, s,
                       inv);
            return cudaGetLastError();
        }
        const bool vec = n % 4 == 0 && (uintptr_t)x % (4 * sizeof(Ti)) == 0 && (uintptr_t)y % (4 * sizeof(To)) == 0;
        if (vec)
            launch_pdl(q8_cast4_kernel<Ti, To>, grid_for(n / 4, 256), 256, 0, st, (const Vec<Ti, 4> *)x,
                       (Vec<To, 4> *)y, n / 4, s, inv);
        else
            launch_pdl(q8_cast_kernel<Ti, To>, grid_for(n, 256), 256, 0, st, (const Ti *)x, (To *)y, n, s, inv);
        return cudaGetLastError();
    }
    // NCHW -> NHWC transposes [N][C][HW]; NHWC -> NCHW transposes [N][HW][C]
    const int64_t hw = sh.h * sh.w;
    const int R = (int)(lay_in == SN_NCHW ? sh.c : hw), C = (int)(lay_in == SN_NCHW ? hw : sh.c);
    if (sh.n > 65535) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)((C + QT - 1) / QT), (unsigned)((R + QT - 1) / QT), (unsigned)sh.n);
    constexpr int SI = (int)sizeof(Ti);
    const int vi = q8_row_vec(C, SI, x), vo = q8_row_vec(R, (int)sizeof(To), y);
    const Ti *xi = (const Ti *)x;
    To *yo = (To *)y;
    if (vi == 16) launch_q8_transpose<Ti, To, 16>(vo, grid, st, xi, yo, R, C, s, inv);
    else if (vi == 8) launch_q8_transpose<Ti, To, 8>(vo, grid, st, xi, yo, R, C, s, inv);
    else if (vi == 4) launch_q8_transpose<Ti, To, (SI <= 4 ? 4 : SI)>(vo, grid, st, xi, yo, R, C, s, inv);
    else launch_q8_transpose<Ti, To, SI>(vo, grid, st, xi, yo, R, C, s, inv);
    return cudaGetLastError();
}

cudaError_t convert_q8(const void *x, int dt_in, int lay_in, void *y, int dt_out, int lay_out, Shape sh,
                       float qscale, cudaStream_t st) {
    if (!(qscale > 0.0f) || !std::isfinite(qscale)) return cudaErrorInvalidValue;
    const float inv = 1.0f / qscale;
    if (dt_in == SN_QI8 && dt_out == SN_QI8)
        return convert_q8_t<int8_t, int8_t>(x, lay_in, y, lay_out, sh, qscale, inv, st);
    if (dt_in == SN_QI8) {
        if (dt_out == SN_F32) return convert_q8_t<int8_t, float>(x, lay_in, y, lay_out, sh, qscale, inv, st);
        if (dt_out == SN_F16) return convert_q8_t<int8_t, __half>(x, lay_in, y, lay_out, sh, qscale, inv, st);
        if (dt_out == SN_BF16)
            return convert_q8_t<int8_t, __nv_bfloat16>(x, lay_in, y, lay_out, sh, qscale, inv, st);
        return cudaErrorInvalidValue;
    }
    if (dt_out != SN_QI8) return cudaErrorInvalidValue;
    if (dt_in == SN_F32) return convert_q8_t<float, int8_t>(x, lay_in, y, lay_out, sh, qscale, inv, st);
    if (dt_in == SN_F16) return convert_q8_t<__half, int8_t>(x, lay_in, y, lay_out, sh, qscale, inv, st);
    if (dt_in == SN_BF16) return convert_q8_t<__nv_bfloat16, int8_t>(x, lay_in, y, lay_out, sh, qscale, inv, st);
    return cudaErrorInvalidValue;
}

// deterministic pseudo-random codes in [-127, 127] (profiling scratch)
__global__ void q8_fill_kernel(int8_t *y, int64_t n, uint32_t seed) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t h = (uint32_t)i * 2654435761u ^ seed;
        h ^= h >> 16;
        h *= 0x7feb352du;
        h ^= h >> 15;
        y[i] = (int8_t)((int)(h % 255u) - 127);
    }
}

cudaError_t fill_q8(void *y, int64_t n, uint32_t seed, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    launch_pdl(q8_fill_kernel, grid_for(n, 256), 256, 0, st, (int8_t *)y, n, seed);
    return cudaGetLastError();
}

// ===========================================================================
// weights: per-output-channel scales, then codes in the routine's format
// ===========================================================================
__global__ void __launch_bounds__(256) q8_wscale_kernel(const float *__restrict__ w, float *__restrict__ scale,
                                                        int64_t per_k) {
    griddep_launch();
    griddep_wait();
    const float *wk = w + blockIdx.x * per_k;
    float m = 0.0f;
    for (int64_t j = threadIdx.x; j < per_k; j += blockDim.x) m = fmaxf(m, fabsf(wk[j]));
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    __shared__ float part[8];
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int i = 1; i < 8; ++i) m = fmaxf(m, part[i]);
        scale[blockIdx.x] = m > 0.0f ? __fdiv_rn(m, (float)QMAX) : 1.0f;
    }
}

// out[i] = code of w[k][c][r][s] for the format's element i
__global__ void q8_wcode_kernel(const float *__restrict__ w, const float *__restrict__ scale, int8_t *__restrict__ out,
                                int fmt, int64_t K, int64_t Cg, int64_t R, int64_t S) {
    griddep_launch();
    griddep_wait();
    const int64_t total = K * Cg * R * S;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int64_t kk, c, r, s;
        if (fmt == W_RSCK) {  // [R][S][Cg][K]
            kk = i % K;
            c = (i / K) % Cg;
            s = (i / (K * Cg)) % S;
            r = i / (K * Cg * S);
        } else if (fmt == W_KRSC) {  // [K][R][S][Cg]
            c = i % Cg;
            s = (i / Cg) % S;
            r = (i / (Cg * S)) % R;
            kk = i / (Cg * S * R);
        } else {  // [K][Cg][R][S]
            s = i % S;
            r = (i / S) % R;
            c = (i / (S * R)) % Cg;
            kk = i / (S * R * Cg);
        }
        const float v = w[((kk * Cg + c) * R + r) * S + s];
        const int q = __float2int_rn(__fdiv_rn(v, scale[kk]));
        out[i] = (int8_t)max(-QMAX, min(QMAX, q));
    }
}

cudaError_t weight_format_q8(const float *w, void *out, int fmt, int64_t K, int64_t Cg, int64_t R, int64_t S,
                             cudaStream_t st) {
    if (fmt != W_KCRS && fmt != W_RSCK && fmt != W_KRSC) return cudaErrorInvalidValue;
    const int64_t elems = K * Cg * R * S;
    float *scale = reinterpret_cast<float *>(static_cast<char *>(out) + align16(elems));
    launch_pdl(q8_wscale_kernel, dim3((unsigned)K), 256, 0, st, w, scale, Cg * R * S);
    launch_pdl(q8_wcode_kernel, grid_for(elems, 256), 256, 0, st, w, (const float *)scale, (int8_t *)out, fmt, K, Cg,
               R, S);
    return cudaGetLastError();
}

// ===========================================================================
// conv2 / dwconv2, direct: one output code per thread (any layout, groups,
// stride, dilation; optional residual)
// ===========================================================================
struct Q8Scales {
    float s_x, s_r, inv_out;
};

template <bool NHWC, typename TO>
__global__ void q8_conv_direct_kernel(const int8_t *__restrict__ x, const int8_t *__restrict__ w,
                                      const float *__restrict__ ws, const float *__restrict__ bias,
                                      const int8_t *__restrict__ res, TO *__restrict__ y, ConvDims d, Q8Scales q) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    const int Cg = d.C / d.groups, Kg = d.K / d.groups;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int kk, p, qq;
        int64_t n;
        if (NHWC) {
            kk = (int)(i % d.K);
            const int64_t pix = i / d.K;
            qq = (int)(pix % d.Q);
            p = (int)((pix / d.Q) % d.P);
            n = pix / ((int64_t)d.Q * d.P);
        } else {
            qq = (int)(i % d.Q);
            p = (int)((i / d.Q) % d.P);
            kk = (int)((i / ((int64_t)d.Q * d.P)) % d.K);
            n = i / ((int64_t)d.Q * d.P * d.K);
        }
        const int c0 = (kk / Kg) * Cg;
        int acc = 0;
        for (int r = 0; r < d.R; ++r) {
            const int h = p * d.sh - d.ph + r * d.dh;
            if (h < 0 || h >= d.H) continue;
            for (int s = 0; s < d.S; ++s) {
                const int ww = qq * d.sw - d.pw + s * d.dw;
                if (ww < 0 || ww >= d.W) continue;
                if (NHWC) {
                    const int8_t *xp = x + (((n * d.H + h) * d.W + ww) * d.C + c0);
                    const int8_t *wp = w + ((int64_t)(r * d.S + s) * Cg) * d.K + kk;  // [R][S][Cg][K]
                    for (int c = 0; c < Cg; ++c) acc += (int)xp[c] * (int)wp[(int64_t)c * d.K];
                } else {
                    for (int c = 0; c < Cg; ++c)
                        acc += (int)x[((n * d.C + c0 + c) * d.H + h) * (int64_t)d.W + ww] *
                               (int)w[(((int64_t)kk * Cg + c) * d.R + r) * d.S + s];  // [K][Cg][R][S]
                }
            }
        }
        const float rv = res ? __fmul_rn((float)res[i], q.s_r) : 0.0f;  // residual: the output's index
        y[i] = q8_out<TO>(q8_value(acc, q.s_x, ws[kk], bias[kk], rv, d.act), q.inv_out);
    }
}

// the schema dtype the routine writes: qint8, or a float type when the
// dequantisation is fused into its epilogue
static int out_dtype(const LaunchArgs &a) { return a.out_schema.dtype < 0 ? a.schema.dtype : a.out_schema.dtype; }

#define SN_Q8_OUT_SWITCH(dt, TO, ...)                               \
    switch (dt) {                                                   \
    case SN_QI8: { using TO = int8_t; __VA_ARGS__; break; }         \
    case SN_F16: { using TO = __half; __VA_ARGS__; break; }         \
    case SN_BF16: { using TO = __nv_bfloat16; __VA_ARGS__; break; } \
    case SN_F32: { using TO = float; __VA_ARGS__; break; }          \
    default: return cudaErrorInvalidValue;                          \
    }

static Q8Scales scales_of(const LaunchArgs &a) {
    return Q8Scales{a.qs_in[0], a.qs_in[1], a.qs_out > 0.0f ? 1.0f / a.qs_out : 0.0f};
}

// the input scales, and the output scale when the output is qint8
static bool scales_ok(const LaunchArgs &a, int n_in) {
    for (int i = 0; i < n_in; ++i)
        if (!(a.qs_in[i] > 0.0f) || !std::isfinite(a.qs_in[i])) return false;
    return out_dtype(a) != SN_QI8 || (a.qs_out > 0.0f && std::isfinite(a.qs_out));
}

cudaError_t q8_conv_direct(const LaunchArgs &a) {
    if (!scales_ok(a, a.in[1] ? 2 : 1)) return cudaErrorInvalidValue;
    const ConvDims d = conv_dims(a);
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    const int64_t elems = (int64_t)d.K * (d.C / d.groups) * d.R * d.S;
    const float *ws = wscales(a.wt, elems);
    SN_Q8_OUT_SWITCH(out_dtype(a), TO, {
        if (a.schema.layout == SN_NHWC)
            launch_pdl(q8_conv_direct_kernel<true, TO>, grid_for(total, 256), 256, 0, a.stream,
                       (const int8_t *)a.in[0], (const int8_t *)a.wt, ws, a.bias, (const int8_t *)a.in[1], (TO *)a.out,
                       d, scales_of(a));
        else
            launch_pdl(q8_conv_direct_kernel<false, TO>, grid_for(total, 256), 256, 0, a.stream,
                       (const int8_t *)a.in[0], (const int8_t *)a.wt, ws, a.bias, (const int8_t *)a.in[1], (TO *)a.out,
                       d, scales_of(a));
    });
    return cudaGetLastError();
}

// ===========================================================================
// conv2, NHWC implicit GEMM with dp4a (groups 1, C % 4 == 0, K % 4 == 0)
// ===========================================================================
// A CTA computes 64 output pixels x 64 output channels.  The reduction runs
// over (r, s, 32-channel chunk) steps; each step stages the 64 pixels' and the
// 64 filters' 32 channel bytes in shared memory as 8 int32 words, word-major,
// and every thread accumulates a 4 x 4 block with dp4a (16 per word).
// Weights are [K][R][S][C].
constexpr int DP_BM = 64, DP_BN = 64, DP_WORDS = 8;

template <typename TO>
__global__ void __launch_bounds__(256) q8_conv_dp4a_kernel(const int8_t *__restrict__ x, const int8_t *__restrict__ w,
                                                           const float *__restrict__ ws,
                                                           const float *__restrict__ bias,
                                                           const int8_t *__restrict__ res, TO *__restrict__ y,
                                                           ConvDims d, Q8Scales q) {
    griddep_launch();
    __shared__ __align__(16) int As[2][DP_WORDS][DP_BM];
    __shared__ __align__(16) int Bs[2][DP_WORDS][DP_BN];
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;  // compute: channels 4*tx.., pixels 4*ty..
    const int64_t M = (int64_t)d.N * d.P * d.Q;
    const int64_t m0 = (int64_t)blockIdx.x * DP_BM;
    const int k0 = blockIdx.y * DP_BN;
    // loader role: pixel / filter lm = tid / 4 of the tile, words 2*(tid%4) and +1
    const int lm = tid >> 2, lw = (tid & 3) * 2;
    const int64_t mpix = m0 + lm;
    const bool pix_ok = mpix < M;
    int pn = 0, pp = 0, pq = 0;
    if (pix_ok) {
        pq = (int)(mpix % d.Q);
        pp = (int)((mpix / d.Q) % d.P);
        pn = (int)(mpix / ((int64_t)d.Q * d.P));
    }
    const int lk = k0 + lm;
    const bool k_ok = lk < d.K;
    griddep_wait();
    int acc[4][4] = {};
    const int chunks = (d.C + 31) / 32;
    const int steps = d.R * d.S * chunks;
    auto load = [&](int step, int buf) {
        const int ch = step % chunks, rs = step / chunks;
        const int r = rs / d.S, s = rs - r * d.S;
        const int h = pp * d.sh - d.ph + r * d.dh, ww = pq * d.sw - d.pw + s * d.dw;
        const bool in_img = pix_ok && h >= 0 && h < d.H && ww >= 0 && ww < d.W;
        const int8_t *xp = x + (((int64_t)pn * d.H + h) * d.W + ww) * d.C;
        const int8_t *wp = w + (((int64_t)lk * d.R + r) * d.S + s) * d.C;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int c = ch * 32 + (lw + e) * 4;
            const bool c_ok = c < d.C;
            As[buf][lw + e][lm] = (in_img && c_ok) ? *reinterpret_cast<const int *>(xp + c) : 0;
            Bs[buf][lw + e][lm] = (k_ok && c_ok) ? *reinterpret_cast<const int *>(wp + c) : 0;
        }
    };
    load(0, 0);
    __syncthreads();
    for (int st = 0; st < steps; ++st) {
        const int buf = st & 1;
        if (st + 1 < steps) load(st + 1, buf ^ 1);
#pragma unroll
        for (int kw = 0; kw < DP_WORDS; ++kw) {
            const int4 av = *reinterpret_cast<const int4 *>(&As[buf][kw][ty * 4]);
            const int4 bv = *reinterpret_cast<const int4 *>(&Bs[buf][kw][tx * 4]);
            const int a4[4] = {av.x, av.y, av.z, av.w}, b4[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = dp4a(a4[i], b4[j], acc[i][j]);
        }
        __syncthreads();
    }
    const int kb = k0 + tx * 4;
    if (kb >= d.K) return;
    float sw[4], bs[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        sw[j] = ws[kb + j];
        bs[j] = bias[kb + j];
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t m = m0 + ty * 4 + i;
        if (m >= M) break;
        char4 rr = make_char4(0, 0, 0, 0);
        if (res) rr = *reinterpret_cast<const char4 *>(res + m * d.K + kb);
        const int8_t r4[4] = {rr.x, rr.y, rr.z, rr.w};
        TO o[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float rv = res ? __fmul_rn((float)r4[j], q.s_r) : 0.0f;
            o[j] = q8_out<TO>(q8_value(acc[i][j], q.s_x, sw[j], bs[j], rv, d.act), q.inv_out);
        }
        if constexpr (std::is_same<TO, int8_t>::value) {
            *reinterpret_cast<char4 *>(y + m * d.K + kb) = make_char4(o[0], o[1], o[2], o[3]);
        } else {
#pragma unroll
            for (int j = 0; j < 4; ++j) y[m * d.K + kb + j] = o[j];
        }
    }
}

bool q8_conv_dp4a_applies(const Layer &l, const Shape &in, sn_schema s) {
    const sn_conv_params &p = l.conv;
    return l.type == SN_L_CONV2 && s.layout == SN_NHWC && p.groups == 1 && in.c % 4 == 0 && p.c_out % 4 == 0 &&
           (int64_t)in.n * l.out.h * l.out.w < ((int64_t)1 << 31) * DP_BM;
}

cudaError_t q8_conv_dp4a(const LaunchArgs &a) {
    if (!scales_ok(a, a.in[1] ? 2 : 1)) return cudaErrorInvalidValue;
    const ConvDims d = conv_dims(a);
    if (d.C % 4 || d.K % 4 || d.groups != 1) return cudaErrorInvalidValue;
    const int64_t M = (int64_t)d.N * d.P * d.Q;
    const int64_t elems = (int64_t)d.K * d.C * d.R * d.S;
    const dim3 grid((unsigned)((M + DP_BM - 1) / DP_BM), (unsigned)((d.K + DP_BN - 1) / DP_BN));
    if (grid.y > 65535) return cudaErrorInvalidValue;
    SN_Q8_OUT_SWITCH(out_dtype(a), TO,
                     launch_pdl(q8_conv_dp4a_kernel<TO>, grid, 256, 0, a.stream, (const int8_t *)a.in[0],
                                (const int8_t *)a.wt, wscales(a.wt, elems), a.bias, (const int8_t *)a.in[1],
                                (TO *)a.out, d, scales_of(a)));
    return cudaGetLastError();
}

// ===========================================================================
// dense: one warp per output feature, NB images per pass over its weight row
// (16-byte loads and dp4a when in_features % 16 == 0)
// ===========================================================================
template <int NB, bool V16, typename TO>
__global__ void __launch_bounds__(256) q8_dense_kernel(const int8_t *__restrict__ x, const int8_t *__restrict__ w,
                                                       const float *__restrict__ ws, const float *__restrict__ bias,
                                                       TO *__restrict__ y, int N, int I, int O, int act,
                                                       Q8Scales q) {
    griddep_launch();
    griddep_wait();
    const int lane = threadIdx.x & 31;
    const int o = blockIdx.x * 8 + (threadIdx.x >> 5);
    if (o >= O) return;
    const int8_t *wr = w + (int64_t)o * I;
    for (int n0 = 0; n0 < N; n0 += NB) {
        int acc[NB] = {};
        if (V16) {
            int i = lane * 16;
            for (; i < I; i += 512) {
                const int4 wv = *reinterpret_cast<const int4 *>(wr + i);
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    if (n0 + b >= N) break;
                    const int4 xv = *reinterpret_cast<const int4 *>(x + (int64_t)(n0 + b) * I + i);
                    acc[b] = dp4a(xv.x, wv.x, acc[b]);
                    acc[b] = dp4a(xv.y, wv.y, acc[b]);
                    acc[b] = dp4a(xv.z, wv.z, acc[b]);
                    acc[b] = dp4a(xv.w, wv.w, acc[b]);
                }
            }
        } else {
            for (int i = lane; i < I; i += 32) {
                const int wv = wr[i];
#pragma unroll
                for (int b = 0; b < NB; ++b)
                    if (n0 + b < N) acc[b] += (int)x[(int64_t)(n0 + b) * I + i] * wv;
            }
        }
#pragma unroll
        for (int b = 0; b < NB; ++b)
            for (int off = 16; off; off >>= 1) acc[b] += __shfl_xor_sync(0xffffffffu, acc[b], off);
        if (lane < NB && n0 + lane < N) {
            int v = acc[0];
#pragma unroll
            for (int b = 1; b < NB; ++b)
                if (lane == b) v = acc[b];
            y[(int64_t)(n0 + lane) * O + o] = q8_out<TO>(q8_value(v, q.s_x, ws[o], bias[o], 0.0f, act), q.inv_out);
        }
    }
}

cudaError_t q8_dense(const LaunchArgs &a) {
    if (!scales_ok(a, 1)) return cudaErrorInvalidValue;
    const Layer &l = *a.layer;
    const int N = (int)a.in_shapes[0].n, I = l.dense_in, O = l.dense_out;
    const float *ws = wscales(a.wt, (int64_t)I * O);
    const dim3 grid((unsigned)((O + 7) / 8));
    const bool v16 = I % 16 == 0 && (uintptr_t)a.in[0] % 16 == 0 && (uintptr_t)a.wt % 16 == 0;
#define SN_Q8_DENSE(NB)                                                                                        \
    SN_Q8_OUT_SWITCH(out_dtype(a), TO,                                                                         \
                     (v16 ? launch_pdl(q8_dense_kernel<NB, true, TO>, grid, 256, 0, a.stream,                  \
                                       (const int8_t *)a.in[0], (const int8_t *)a.wt, ws, a.bias, (TO *)a.out, \
                                       N, I, O, l.act, scales_of(a))                                           \
                          : launch_pdl(q8_dense_kernel<NB, false, TO>, grid, 256, 0, a.stream,                 \
                                       (const int8_t *)a.in[0], (const int8_t *)a.wt, ws, a.bias, (TO *)a.out, \
                                       N, I, O, l.act, scales_of(a))))
    if (N <= 1) {
        SN_Q8_DENSE(1);
    } else if (N <= 2) {
        SN_Q8_DENSE(2);
    } else if (N <= 4) {
        SN_Q8_DENSE(4);
    } else {
        SN_Q8_DENSE(8);
    }
#undef SN_Q8_DENSE
    return cudaGetLastError();
}

// ===========================================================================
// max pool, global average pool, add, squeeze-and-excite scale
// ===========================================================================
template <bool NHWC, typename TO>
__global__ void q8_maxpool_kernel(const int8_t *__restrict__ x, TO *__restrict__ y, int N, int C, int H, int W,
                                  int P, int Q, sn_pool_params pp, float s_x, float inv) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)N * C * P * Q;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int c, p, q;
        int64_t n;
        if (NHWC) {
            c = (int)(i % C);
            q = (int)((i / C) % Q);
            p = (int)((i / ((int64_t)C * Q)) % P);
            n = i / ((int64_t)C * Q * P);
        } else {
            q = (int)(i % Q);
            p = (int)((i / Q) % P);
            c = (int)((i / ((int64_t)Q * P)) % C);
            n = i / ((int64_t)Q * P * C);
        }
        int m = -(1 << 20);  // below every code: padding never wins
        for (int r = 0; r < pp.kh; ++r) {
            const int h = p * pp.sh - pp.ph + r;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < pp.kw; ++s) {
                const int ww = q * pp.sw - pp.pw + s;
                if (ww < 0 || ww >= W) continue;
                const int64_t xi = NHWC ? ((n * H + h) * W + ww) * C + c : ((n * C + c) * H + h) * (int64_t)W + ww;
                m = max(m, (int)x[xi]);
            }
        }
        y[i] = q8_out<TO>(__fmul_rn((float)m, s_x), inv);
    }
}

cudaError_t q8_maxpool(const LaunchArgs &a) {
    if (!scales_ok(a, 1)) return cudaErrorInvalidValue;
    const Shape &i = a.in_shapes[0], &o = a.layer->out;
    const int64_t total = o.numel();
    const float inv = scales_of(a).inv_out;
    SN_Q8_OUT_SWITCH(out_dtype(a), TO, {
        if (a.schema.layout == SN_NHWC)
            launch_pdl(q8_maxpool_kernel<true, TO>, grid_for(total, 256), 256, 0, a.stream, (const int8_t *)a.in[0],
                       (TO *)a.out, (int)i.n, (int)i.c, (int)i.h, (int)i.w, (int)o.h, (int)o.w, a.layer->pool,
                       a.qs_in[0], inv);
        else
            launch_pdl(q8_maxpool_kernel<false, TO>, grid_for(total, 256), 256, 0, a.stream,
                       (const int8_t *)a.in[0], (TO *)a.out, (int)i.n, (int)i.c, (int)i.h, (int)i.w, (int)o.h,
                       (int)o.w, a.layer->pool, a.qs_in[0], inv);
    });
    return cudaGetLastError();
}

// NCHW: one warp per (n, c) plane; NHWC: one thread per (n, c), consecutive
// threads on consecutive channels.  The code sum is exact; its value is
// (float(sum) * s_x) / (H*W), two roundings.
template <bool NHWC, typename TO>
__global__ void q8_gap_kernel(const int8_t *__restrict__ x, TO *__restrict__ y, int N, int C, int HW, float s_x,
                              float inv) {
    griddep_launch();
    griddep_wait();
    if (NHWC) {
        for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < (int64_t)N * C;
             t += (int64_t)gridDim.x * blockDim.x) {
            const int64_t n = t / C;
            const int c = (int)(t % C);
            int sum = 0;
            for (int j = 0; j < HW; ++j) sum += x[(n * HW + j) * C + c];
            y[t] = q8_out<TO>(__fdiv_rn(__fmul_rn(__int2float_rn(sum), s_x), (float)HW), inv);
        }
    } else {
        const int lane = threadIdx.x & 31;
        const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
        for (int64_t t = blockIdx.x * (int64_t)(blockDim.x >> 5) + (threadIdx.x >> 5); t < (int64_t)N * C;
             t += warps) {
            int sum = 0;
            for (int j = lane; j < HW; j += 32) sum += x[t * HW + j];
            for (int off = 16; off; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
            if (lane == 0) y[t] = q8_out<TO>(__fdiv_rn(__fmul_rn(__int2float_rn(sum), s_x), (float)HW), inv);
        }
    }
}

cudaError_t q8_gap(const LaunchArgs &a) {
    if (!scales_ok(a, 1)) return cudaErrorInvalidValue;
    const Shape &i = a.in_shapes[0];
    const float inv = scales_of(a).inv_out;
    const int64_t nc = i.n * i.c;
    if (i.h * i.w >= (1 << 23)) return cudaErrorInvalidValue;  // int32 sums stay exact
    SN_Q8_OUT_SWITCH(out_dtype(a), TO, {
        if (a.schema.layout == SN_NHWC)
            launch_pdl(q8_gap_kernel<true, TO>, grid_for(nc, 256), 256, 0, a.stream, (const int8_t *)a.in[0],
                       (TO *)a.out, (int)i.n, (int)i.c, (int)(i.h * i.w), a.qs_in[0], inv);
        else
            launch_pdl(q8_gap_kernel<false, TO>, grid_for(nc * 32, 256), 256, 0, a.stream, (const int8_t *)a.in[0],
                       (TO *)a.out, (int)i.n, (int)i.c, (int)(i.h * i.w), a.qs_in[0], inv);
    });
    return cudaGetLastError();
}

// MUL = false: y = act(a * s_a + b * s_b); MUL = true: y = act((a * s_a) *
// (b[n, c] * s_b)), b an N x C blob
template <bool MUL, bool NHWC, typename TO>
__global__ void q8_binary_kernel(const int8_t *__restrict__ a, const int8_t *__restrict__ b, TO *__restrict__ y,
                                 int64_t total, int C, int64_t HW, float s_a, float s_b, int act, float inv) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float va = __fmul_rn((float)a[i], s_a);
        float v;
        if (MUL) {
            const int64_t n = i / (HW * C);
            const int c = NHWC ? (int)(i % C) : (int)((i / HW) % C);
            v = __fmul_rn(va, __fmul_rn((float)b[n * C + c], s_b));
        } else {
            v = __fadd_rn(va, __fmul_rn((float)b[i], s_b));
        }
        y[i] = q8_out<TO>(q8_act(v, act), inv);
    }
}

template <bool MUL>
static cudaError_t q8_binary(const LaunchArgs &a) {
    if (!scales_ok(a, 2)) return cudaErrorInvalidValue;
    const Shape &o = a.layer->out;
    const int64_t total = o.numel();
    const float inv = scales_of(a).inv_out;
    const int act = a.layer->act;
    SN_Q8_OUT_SWITCH(out_dtype(a), TO, {
        if (a.schema.layout == SN_NHWC)
            launch_pdl(q8_binary_kernel<MUL, true, TO>, grid_for(total, 256), 256, 0, a.stream,
                       (const int8_t *)a.in[0], (const int8_t *)a.in[1], (TO *)a.out, total, (int)o.c, o.h * o.w,
                       a.qs_in[0], a.qs_in[1], act, inv);
        else
            launch_pdl(q8_binary_kernel<MUL, false, TO>, grid_for(total, 256), 256, 0, a.stream,
                       (const int8_t *)a.in[0], (const int8_t *)a.in[1], (TO *)a.out, total, (int)o.c, o.h * o.w,
                       a.qs_in[0], a.qs_in[1], act, inv);
    });
    return cudaGetLastError();
}

cudaError_t q8_add(const LaunchArgs &a) { return q8_binary<false>(a); }
cudaError_t q8_mul(const LaunchArgs &a) { return q8_binary<true>(a); }

// ===========================================================================
// calibration: running max |x| of a blob (as fp32 bits; non-negative floats
// order like their bit patterns)
// ===========================================================================
template <typename T>
__global__ void absmax_kernel(const T *__restrict__ x, int64_t n, unsigned *__restrict__ out) {
    griddep_launch();
    griddep_wait();
    float m = 0.0f;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        m = fmaxf(m, fabsf(ldf<T>(x + i)));
    for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    if ((threadIdx.x & 31) == 0) atomicMax(out, __float_as_uint(m));
}

cudaError_t absmax(const void *x, int dt, int64_t n, unsigned *out, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (dt == SN_QI8) return cudaErrorInvalidValue;
    SN_DT_SWITCH(dt, T, launch_pdl(absmax_kernel<T>, grid_for(n, 256, 152LL * 8), 256, 0, st, (const T *)x, n, out));
    return cudaGetLastError();
}

}  // namespace k
}  // namespace sn
