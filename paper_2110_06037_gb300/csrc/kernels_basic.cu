// Adapt conversion, weight formatting, direct convolution, depthwise
// convolution, pooling, elementwise add and dense routines (CUDA cores).
#include <algorithm>
#include <type_traits>

#include "kern_common.cuh"

namespace sn {
namespace k {

__device__ int g_error_word = 0;

int *device_error_word() {
    void *p = nullptr;
    cudaGetSymbolAddress(&p, g_error_word);
    return static_cast<int *>(p);
}

// ===========================================================================
// adapt: layout permutation and/or RNE cast (section III-C, jobs 2 and 3)
// ===========================================================================

// same layout: elementwise cast (or copy)
template <typename Ti, typename To>
__global__ void cast_kernel(const Ti *__restrict__ x, To *__restrict__ y, int64_t n) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        stf<To>(y + i, ldf<Ti>(x + i));
}

// VB-byte vector access to VB / sizeof(T) consecutive elements, as floats
template <typename T, int VB>
struct VecIO {
    static constexpr int E = VB / (int)sizeof(T);
    using V = typename std::conditional<
        VB == 16, uint4,
        typename std::conditional<VB == 8, uint2,
                                  typename std::conditional<VB == 4, uint32_t, uint16_t>::type>::type>::type;
    __device__ __forceinline__ static void load(const T *p, float (&f)[E]) {
        const V v = *reinterpret_cast<const V *>(p);
        const T *t = reinterpret_cast<const T *>(&v);
#pragma unroll
        for (int e = 0; e < E; ++e) f[e] = ldf<T>(t + e);
    }
    __device__ __forceinline__ static void store(T *p, const float (&f)[E]) {
        V v;
        T *t = reinterpret_cast<T *>(&v);
#pragma unroll
        for (int e = 0; e < E; ++e) t[e] = cvt<T>(f[e]);
        *reinterpret_cast<V *>(p) = v;
    }
};

// same layout, 8 elements per thread and iteration with 16-byte accesses
// (n % 8 == 0, 16-byte aligned bases)
template <typename Ti, typename To>
__global__ void cast_vec8_kernel(const Ti *__restrict__ x, To *__restrict__ y, int64_t n8) {
    griddep_launch();
    griddep_wait();
    constexpr int EI = VecIO<Ti, 16>::E, EO = VecIO<To, 16>::E;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
         i += (int64_t)gridDim.x * blockDim.x) {
        float f[8];
#pragma unroll
        for (int j = 0; j < 8; j += EI) {
            float g[EI];
            VecIO<Ti, 16>::load(x + i * 8 + j, g);
#pragma unroll
            for (int e = 0; e < EI; ++e) f[j + e] = g[e];
        }
#pragma unroll
        for (int j = 0; j < 8; j += EO) {
            float g[EO];
#pragma unroll
            for (int e = 0; e < EO; ++e) g[e] = f[j + e];
            VecIO<To, 16>::store(y + i * 8 + j, g);
        }
    }
}

// 16-byte vectorised copy when dtypes match
__global__ void copy16_kernel(const uint4 *__restrict__ x, uint4 *__restrict__ y, int64_t n16) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16;
         i += (int64_t)gridDim.x * blockDim.x)
        y[i] = x[i];
}

// batched transpose y[b][c][r] = x[b][r][c] with a cast, through a 64x64
// shared-memory tile: VBI-byte vectors along the input rows, VBO-byte vectors
// along the output rows (the widest the row lengths and bases allow: a
// 14 x 14 plane is 392 bytes of bf16, so its rows take 8-byte vectors)
constexpr int TT = 64;
template <typename Ti, typename To, int VBI, int VBO>
__global__ void __launch_bounds__(256) transpose_vec_kernel(const Ti *__restrict__ x, To *__restrict__ y,
                                                             int64_t R, int64_t Cc) {
    griddep_launch();
    griddep_wait();
    using LI = VecIO<Ti, VBI>;
    using LO = VecIO<To, VBO>;
    constexpr int EI = LI::E, EO = LO::E;
    __shared__ float tile[TT][TT + 1];
    const int64_t b = blockIdx.z;
    const int64_t r0 = (int64_t)blockIdx.y * TT, c0 = (int64_t)blockIdx.x * TT;
    const Ti *xb = x + b * R * Cc;
    To *yb = y + b * R * Cc;
    constexpr int VI = TT / EI;  // input vectors per tile row
#pragma unroll 4
    for (int i = threadIdx.x; i < TT * VI; i += 256) {
        const int row = i / VI, cv = i % VI;
        const int64_t r = r0 + row, c = c0 + cv * EI;
        if (r < R && c < Cc) {
            float f[EI];
            LI::load(xb + r * Cc + c, f);
#pragma unroll
            for (int e = 0; e < EI; ++e) tile[row][cv * EI + e] = f[e];
        }
    }
    __syncthreads();
    constexpr int VO = TT / EO;  // output vectors per tile row (output row = input column)
#pragma unroll 4
    for (int i = threadIdx.x; i < TT * VO; i += 256) {
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

// widest vector (16, 8 or element bytes) that a row of n elements of es bytes
// starting at every row of an aligned base admits
static int row_vec_bytes(int64_t n, int es, const void *base) {
    for (int vb : {16, 8})
        if ((n * es) % vb == 0 && (uintptr_t)base % vb == 0) return vb;
    return es;
}

// few channels (C <= 16): one thread per pixel moves all of its channels;
// the planar side is read/written coalesced across threads, the interleaved
// side as C consecutive elements per thread (C * 32 contiguous per warp).
// Grid: y = image, x = pixels of the image (no index division).
template <typename Ti, typename To, bool TO_NHWC>
__global__ void permute_small_c_kernel(const Ti *__restrict__ x, To *__restrict__ y, int N, int C, int HW) {
    griddep_launch();
    griddep_wait();
    for (int n = blockIdx.y; n < N; n += gridDim.y)
        for (int hw = blockIdx.x * blockDim.x + threadIdx.x; hw < HW; hw += gridDim.x * blockDim.x) {
            const size_t planar0 = (size_t)n * C * HW + hw, inter0 = ((size_t)n * HW + hw) * C;
            for (int c = 0; c < C; ++c) {
                const size_t planar = planar0 + (size_t)c * HW, inter = inter0 + c;
                if (TO_NHWC) stf<To>(y + inter, ldf<Ti>(x + planar));
                else stf<To>(y + planar, ldf<Ti>(x + inter));
            }
        }
}

template <typename Ti, typename To>
static cudaError_t convert_t(const void *x, int lay_in, void *y, int lay_out, Shape s,
                             cudaStream_t st) {
    const int64_t n = s.numel();
    if (n == 0) return cudaSuccess;
    if (lay_in == lay_out || (s.h * s.w == 1) || s.c == 1) {
        if (std::is_same<Ti, To>::value) {
            const int64_t bytes = n * (int64_t)sizeof(Ti);
            if (bytes % 16 == 0 && ((uintptr_t)x % 16) == 0 && ((uintptr_t)y % 16) == 0) {
                launch_pdl(copy16_kernel, grid_for(bytes / 16, 256), 256, 0, st, (const uint4 *)x, (uint4 *)y,
                                                                          bytes / 16);
                return cudaGetLastError();
            }
            return cudaMemcpyAsync(y, x, bytes, cudaMemcpyDeviceToDevice, st);
        }
        if (n % 8 == 0 && ((uintptr_t)x % 16) == 0 && ((uintptr_t)y % 16) == 0)
            launch_pdl(cast_vec8_kernel<Ti, To>, grid_for(n / 8, 256), 256, 0, st, (const Ti *)x, (To *)y, n / 8);
        else
            launch_pdl(cast_kernel<Ti, To>, grid_for(n, 256), 256, 0, st, (const Ti *)x, (To *)y, n);
        return cudaGetLastError();
    }
    if (s.c <= 16) {
        const int64_t HW = s.h * s.w;
        if (HW >= ((int64_t)1 << 31) || s.n >= ((int64_t)1 << 31)) return cudaErrorInvalidValue;
        const dim3 g((unsigned)std::min<int64_t>((HW + 255) / 256, 1024), (unsigned)std::min<int64_t>(s.n, 65535));
        if (lay_in == SN_NCHW)
            launch_pdl(permute_small_c_kernel<Ti, To, true>, g, 256, 0, st, (const Ti *)x, (To *)y, (int)s.n, (int)s.c,
                       (int)HW);
        else
            launch_pdl(permute_small_c_kernel<Ti, To, false>, g, 256, 0, st, (const Ti *)x, (To *)y, (int)s.n,
                       (int)s.c, (int)HW);
        return cudaGetLastError();
    }
    // NCHW -> NHWC: per image [C][HW] -> [HW][C]; NHWC -> NCHW: [HW][C] -> [C][HW]
    const int64_t R = (lay_in == SN_NCHW) ? s.c : s.h * s.w;
    const int64_t Cc = (lay_in == SN_NCHW) ? s.h * s.w : s.c;
    if (s.n > 65535) return cudaErrorInvalidValue;
    dim3 grid((unsigned)((Cc + TT - 1) / TT), (unsigned)((R + TT - 1) / TT), (unsigned)s.n);
    if (grid.y > 65535) return cudaErrorInvalidValue;
    constexpr int SI = (int)sizeof(Ti), SO = (int)sizeof(To);
    const int vi = row_vec_bytes(Cc, SI, x), vo = row_vec_bytes(R, SO, y);
    const Ti *xi = (const Ti *)x;
    To *yo = (To *)y;
#define SN_TRANSPOSE(A, B) launch_pdl(transpose_vec_kernel<Ti, To, A, B>, grid, 256, 0, st, xi, yo, R, Cc)
    if (vi == 16 && vo == 16) SN_TRANSPOSE(16, 16);
    else if (vi == 16 && vo == 8) SN_TRANSPOSE(16, 8);
    else if (vi == 8 && vo == 16) SN_TRANSPOSE(8, 16);
    else if (vi == 16) SN_TRANSPOSE(16, SO);
    else if (vo == 16) SN_TRANSPOSE(SI, 16);
    else SN_TRANSPOSE(SI, SO);
#undef SN_TRANSPOSE
    return cudaGetLastError();
}

cudaError_t convert(const void *x, int dt_in, int lay_in, void *y, int dt_out, int lay_out, Shape s,
                    cudaStream_t st) {
    if (dt_in == SN_QI8 || dt_out == SN_QI8) return cudaErrorInvalidValue;  // needs a scale: convert_q8
    SN_DT_SWITCH(dt_in, Ti, SN_DT_SWITCH(dt_out, To, return convert_t<Ti, To>(x, lay_in, y, lay_out, s, st)));
    return cudaErrorInvalidValue;
}

// deterministic pseudo-random fill in [-scale, scale)
template <typename T>
__global__ void fill_kernel(T *y, int64_t n, uint32_t seed, float scale) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t h = (uint32_t)i * 2654435761u ^ seed;
        h ^= h >> 16;
        h *= 0x7feb352du;
        h ^= h >> 15;
        h *= 0x846ca68bu;
        h ^= h >> 16;
        const float u = (float)(h >> 8) * (1.0f / 16777216.0f);
        stf<T>(y + i, scale * (2.0f * u - 1.0f));
    }
}

cudaError_t fill_pattern(void *y, int dt, int64_t n, uint32_t seed, float scale, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (dt == SN_QI8) return fill_q8(y, n, seed, st);
    SN_DT_SWITCH(dt, T, launch_pdl(fill_kernel<T>, grid_for(n, 256), 256, 0, st, (T *)y, n, seed, scale));
    return cudaGetLastError();
}

// ===========================================================================
// weight formats (from fp32 [K][Cg][R][S])
// ===========================================================================
template <typename T>
__global__ void weight_perm_kernel(const float *__restrict__ w, T *__restrict__ out, int fmt,
                                   int64_t K, int64_t Cg, int64_t R, int64_t S) {
    griddep_launch();
    griddep_wait();
    const int64_t total = K * Cg * R * S;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        // i indexes the source [k][c][r][s]
        const int64_t s = i % S, r = (i / S) % R, c = (i / (S * R)) % Cg, kk = i / (S * R * Cg);
        int64_t o;
        if (fmt == W_KCRS) o = i;
        else if (fmt == W_RSCK) o = ((r * S + s) * Cg + c) * K + kk;
        else if (fmt == W_KRSC_PAD64) o = kk * ((Cg * R * S + 63) / 64 * 64) + (r * S + s) * Cg + c;
        else if (fmt == W_S2D)  // [K][A][4 pixels][16], A = 2 (R <= 4) or 4 tap rows (the rest zero):
            // tap (r, s) -> row r/2, pixel s/2, slot (2(r%2)+s%2)Cg+c
            o = (kk * (R <= 4 ? 2 : 4) + r / 2) * 64 + (s / 2) * 16 + ((r % 2) * 2 + s % 2) * Cg + c;
        else o = ((kk * R + r) * S + s) * Cg + c;  // W_KRSC
        stf<T>(out + o, w[i]);
    }
}

// Winograd F(2x2,3x3) filter transform U = G g G^T (Lavin & Gray), stored
// [16][K][C] so that every xi = 4*a + b is a K x C row-major matrix.
template <typename T>
__global__ void weight_wino_kernel(const float *__restrict__ w, T *__restrict__ out, int64_t K,
                                   int64_t C) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < K * C;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float *g = w + i * 9;  // [3][3] for (k, c) = (i / C, i % C)
        float t[4][3];               // G g
        for (int j = 0; j < 3; ++j) {
            const float g0 = g[0 * 3 + j], g1 = g[1 * 3 + j], g2 = g[2 * 3 + j];
            t[0][j] = g0;
            t[1][j] = 0.5f * (g0 + g1 + g2);
            t[2][j] = 0.5f * (g0 - g1 + g2);
            t[3][j] = g2;
        }
        for (int a = 0; a < 4; ++a) {  // (G g) G^T
            const float h0 = t[a][0], h1 = t[a][1], h2 = t[a][2];
            const float u[4] = {h0, 0.5f * (h0 + h1 + h2), 0.5f * (h0 - h1 + h2), h2};
            for (int b = 0; b < 4; ++b) stf<T>(out + (int64_t)(a * 4 + b) * K * C + i, u[b]);
        }
    }
}

// Winograd F(4x4,3x3) filter transform U = G g G^T with Lavin & Gray's 6x3
// G (points 0, +-1, +-2, infinity), fp32 [36][K][C]
__device__ __forceinline__ void wino4_g(float g0, float g1, float g2, float (&u)[6]) {
    u[0] = 0.25f * g0;
    u[1] = -(g0 + g1 + g2) / 6.f;
    u[2] = -(g0 - g1 + g2) / 6.f;
    u[3] = g0 / 24.f + g1 / 12.f + g2 / 6.f;
    u[4] = g0 / 24.f - g1 / 12.f + g2 / 6.f;
    u[5] = g2;
}
__global__ void weight_wino4_kernel(const float *__restrict__ w, float *__restrict__ out, int64_t K, int64_t C) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < K * C;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float *g = w + i * 9;  // [3][3] for (k, c) = (i / C, i % C)
        float t[6][3];               // G g, column by column
        for (int j = 0; j < 3; ++j) {
            float u[6];
            wino4_g(g[0 * 3 + j], g[1 * 3 + j], g[2 * 3 + j], u);
            for (int a = 0; a < 6; ++a) t[a][j] = u[a];
        }
        for (int a = 0; a < 6; ++a) {  // (G g) G^T
            float u[6];
            wino4_g(t[a][0], t[a][1], t[a][2], u);
            for (int b = 0; b < 6; ++b) out[(int64_t)(a * 6 + b) * K * C + i] = u[b];
        }
    }
}

// Winograd F(6x6,3x3) filter transform U = G g G^T with the 8x3 G of the
// points 0, +-1, +-2, +-1/2 and infinity, fp32 [64][K][C]
__device__ __forceinline__ void wino6_g(float g0, float g1, float g2, float (&u)[8]) {
    u[0] = g0;
    u[1] = -2.f * (g0 + g1 + g2) / 9.f;
    u[2] = -2.f * (g0 - g1 + g2) / 9.f;
    u[3] = g0 / 90.f + g1 / 45.f + 2.f * g2 / 45.f;
    u[4] = g0 / 90.f - g1 / 45.f + 2.f * g2 / 45.f;
    u[5] = 32.f * g0 / 45.f + 16.f * g1 / 45.f + 8.f * g2 / 45.f;
    u[6] = 32.f * g0 / 45.f - 16.f * g1 / 45.f + 8.f * g2 / 45.f;
    u[7] = g2;
}
__global__ void weight_wino6_kernel(const float *__restrict__ w, float *__restrict__ out, int64_t K, int64_t C) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < K * C;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float *g = w + i * 9;  // [3][3] for (k, c) = (i / C, i % C)
        float t[8][3];               // G g, column by column
        for (int j = 0; j < 3; ++j) {
            float u[8];
            wino6_g(g[0 * 3 + j], g[1 * 3 + j], g[2 * 3 + j], u);
            for (int a = 0; a < 8; ++a) t[a][j] = u[a];
        }
        for (int a = 0; a < 8; ++a) {  // (G g) G^T
            float u[8];
            wino6_g(t[a][0], t[a][1], t[a][2], u);
            for (int b = 0; b < 8; ++b) out[(int64_t)(a * 8 + b) * K * C + i] = u[b];
        }
    }
}

cudaError_t weight_format(const float *w, void *out, int fmt, int dt, int64_t K, int64_t Cg,
                          int64_t R, int64_t S, cudaStream_t st) {
    if (dt == SN_QI8) return cudaErrorInvalidValue;  // codes and scales: weight_format_q8
    if (fmt == W_WINO4) {  // fp32 whatever the schema's dtype
        if (R != 3 || S != 3) return cudaErrorInvalidValue;
        launch_pdl(weight_wino4_kernel, grid_for(K * Cg, 256), 256, 0, st, w, (float *)out, K, Cg);
        return cudaGetLastError();
    }
    if (fmt == W_WINO6) {  // fp32 whatever the schema's dtype
        if (R != 3 || S != 3) return cudaErrorInvalidValue;
        launch_pdl(weight_wino6_kernel, grid_for(K * Cg, 256), 256, 0, st, w, (float *)out, K, Cg);
        return cudaGetLastError();
    }
    if (fmt == W_WINO) {
        if (R != 3 || S != 3) return cudaErrorInvalidValue;
        SN_DT_SWITCH(dt, T, launch_pdl(weight_wino_kernel<T>, grid_for(K * Cg, 256), 256, 0, st, w, (T *)out, K, Cg));
        return cudaGetLastError();
    }
    if (fmt == W_KRSC_PAD64) {  // rows padded with zeros to a multiple of 64 taps
        const int64_t kpad = (Cg * R * S + 63) / 64 * 64;
        cudaError_t e = cudaMemsetAsync(out, 0, (size_t)K * kpad * dtype_size(dt), st);
        if (e != cudaSuccess) return e;
    }
    if (fmt == W_S2D) {  // taps outside the kernel and channels past 4 Cg are zero
        if (R > 8 || S > 8 || 4 * Cg > 16) return cudaErrorInvalidValue;
        cudaError_t e = cudaMemsetAsync(out, 0, (size_t)K * (R <= 4 ? 2 : 4) * 64 * dtype_size(dt), st);
        if (e != cudaSuccess) return e;
    }
    SN_DT_SWITCH(dt, T,
                 launch_pdl(weight_perm_kernel<T>, grid_for(K * Cg * R * S, 256), 256, 0, st, w, (T *)out, fmt, K, Cg, R, S));
    return cudaGetLastError();
}

// ===========================================================================
// direct convolution: one output element per thread (the untuned baseline)
// ===========================================================================
template <typename T>
__global__ void conv_direct_nchw(const T *__restrict__ x, const T *__restrict__ w,
                                 const float *__restrict__ bias, const T *__restrict__ res, T *__restrict__ y,
                                 ConvDims d) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    const int Cg = d.C / d.groups, Kg = d.K / d.groups;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int q = (int)(i % d.Q), p = (int)((i / d.Q) % d.P);
        const int kk = (int)((i / ((int64_t)d.Q * d.P)) % d.K);
        const int64_t n = i / ((int64_t)d.Q * d.P * d.K);
        const int c0 = (kk / Kg) * Cg;
        float acc = 0.f;
        for (int c = 0; c < Cg; ++c) {
            const T *xc = x + ((n * d.C + c0 + c) * d.H) * (int64_t)d.W;
            const T *wc = w + ((int64_t)kk * Cg + c) * d.R * d.S;
            for (int r = 0; r < d.R; ++r) {
                const int h = p * d.sh - d.ph + r * d.dh;
                if (h < 0 || h >= d.H) continue;
                for (int s = 0; s < d.S; ++s) {
                    const int ww = q * d.sw - d.pw + s * d.dw;
                    if (ww < 0 || ww >= d.W) continue;
                    acc += ldf<T>(xc + (int64_t)h * d.W + ww) * ldf<T>(wc + r * d.S + s);
                }
            }
        }
        if (res) acc += ldf<T>(res + i);  // residual: same layout and index as the output
        stf<T>(y + i, act_apply(acc + bias[kk], d.act));
    }
}

template <typename T>
__global__ void conv_direct_nhwc(const T *__restrict__ x, const T *__restrict__ w,
                                 const float *__restrict__ bias, const T *__restrict__ res, T *__restrict__ y,
                                 ConvDims d) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    const int Cg = d.C / d.groups, Kg = d.K / d.groups;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int kk = (int)(i % d.K);
        const int64_t pix = i / d.K;
        const int q = (int)(pix % d.Q), p = (int)((pix / d.Q) % d.P);
        const int64_t n = pix / ((int64_t)d.Q * d.P);
        const int c0 = (kk / Kg) * Cg;
        float acc = 0.f;
        for (int r = 0; r < d.R; ++r) {
            const int h = p * d.sh - d.ph + r * d.dh;
            if (h < 0 || h >= d.H) continue;
            for (int s = 0; s < d.S; ++s) {
                const int ww = q * d.sw - d.pw + s * d.dw;
                if (ww < 0 || ww >= d.W) continue;
                const T *xp = x + (((n * d.H + h) * d.W + ww) * d.C + c0);
                const T *wp = w + ((int64_t)(r * d.S + s) * Cg) * d.K + kk;  // [R][S][Cg][K]
                for (int c = 0; c < Cg; ++c) acc += ldf<T>(xp + c) * ldf<T>(wp + (int64_t)c * d.K);
            }
        }
        if (res) acc += ldf<T>(res + i);  // residual: same layout and index as the output
        stf<T>(y + i, act_apply(acc + bias[kk], d.act));
    }
}

cudaError_t conv_direct(const LaunchArgs &a) {
    const ConvDims d = conv_dims(a);
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (a.schema.layout == SN_NCHW)
            launch_pdl(conv_direct_nchw<T>, grid_for(total, 256), 256, 0, a.stream, 
                (const T *)a.in[0], (const T *)a.wt, a.bias, (const T *)a.in[1], (T *)a.out, d);
        else
            launch_pdl(conv_direct_nhwc<T>, grid_for(total, 256), 256, 0, a.stream, 
                (const T *)a.in[0], (const T *)a.wt, a.bias, (const T *)a.in[1], (T *)a.out, d);
    });
    return cudaGetLastError();
}

// ===========================================================================
// depthwise convolution
// ===========================================================================
template <typename T>
__global__ void dw_nhwc(const T *__restrict__ x, const T *__restrict__ w, const float *__restrict__ bias,
                        T *__restrict__ y, ConvDims d) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % d.C);
        const int64_t pix = i / d.C;
        const int q = (int)(pix % d.Q), p = (int)((pix / d.Q) % d.P);
        const int64_t n = pix / ((int64_t)d.Q * d.P);
        float acc = 0.f;
        for (int r = 0; r < d.R; ++r) {
            const int h = p * d.sh - d.ph + r * d.dh;
            if (h < 0 || h >= d.H) continue;
            for (int s = 0; s < d.S; ++s) {
                const int ww = q * d.sw - d.pw + s * d.dw;
                if (ww < 0 || ww >= d.W) continue;
                acc += ldf<T>(x + ((n * d.H + h) * d.W + ww) * d.C + c) *
                       ldf<T>(w + (int64_t)(r * d.S + s) * d.C + c);
            }
        }
        stf<T>(y + i, act_apply(acc + bias[c], d.act));
    }
}

// NHWC, 16 bytes of channels (E lanes) per thread and QB consecutive output
// columns: each input vector a thread needs for its QB outputs is loaded from
// global once per (tap row, column) and reused through L1 by its neighbours;
// weights are [R][S][C].
// acc[e] += x[e] * w[e] over the 16 bytes of x and w (E = 16 / sizeof(T)
// lanes); 16-bit types use the mixed-precision FMA, which equals converting
// both factors to f32 first
template <typename T, int E>
__device__ __forceinline__ void fma16(float (&acc)[E], const uint4 &x, const uint4 &w) {
    if constexpr (sizeof(T) == 2) {
        mac2<T>(acc[0], acc[1], x.x, w.x);
        mac2<T>(acc[2], acc[3], x.y, w.y);
        mac2<T>(acc[4], acc[5], x.z, w.z);
        mac2<T>(acc[6], acc[7], x.w, w.w);
    } else {
        const T *xp = reinterpret_cast<const T *>(&x);
        const T *wp = reinterpret_cast<const T *>(&w);
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] = fmaf(ldf<T>(xp + e), ldf<T>(wp + e), acc[e]);
    }
}

// One thread: QB consecutive output columns x E channels (16 bytes) of one
// output row.  The grid's y axis walks the N x P output rows, its x axis the
// (column block, channel vector) pairs of a row with the channel vector
// fastest (coalesced 16-byte accesses); all index math is 32-bit, one
// division per thread (64-bit division and modulo by runtime values cost
// more than the arithmetic of the taps).
template <typename T, int QB, int SW>  // SW = 1 or 2: 3x3 fast path for that stride; 0 = any
__global__ void __launch_bounds__(256, 2) dw_nhwc_vec(const T *__restrict__ x, const T *__restrict__ w,
                                                      const float *__restrict__ bias, T *__restrict__ y, ConvDims d,
                                                      int CV, int QBLK) {
    griddep_launch();
    griddep_wait();
    constexpr int E = 16 / sizeof(T);
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= QBLK * CV) return;
    const int qb = t / CV, cv = t - qb * CV;
    const int c0 = cv * E, q0 = qb * QB;
    float b[E];
    {
        const float4 b0 = *reinterpret_cast<const float4 *>(bias + c0);
        const float4 b1 = *reinterpret_cast<const float4 *>(bias + c0 + 4);
        const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
        for (int e = 0; e < E; ++e) b[e] = bb[e];
    }
    for (int rowi = blockIdx.y; rowi < d.N * d.P; rowi += gridDim.y) {
        const int n = rowi / d.P, p = rowi - n * d.P;
        if constexpr (std::is_same<T, __half>::value && SW > 0) {
            // fp16 3x3: packed half2 multiply-adds accumulating in fp16, in the
            // same order as the ring kernel (bias, rows, columns)
            __half2 hacc[QB][4];
#pragma unroll
            for (int j = 0; j < QB; ++j)
#pragma unroll
                for (int k = 0; k < 4; ++k) hacc[j][k] = __floats2half2_rn(b[2 * k], b[2 * k + 1]);
            constexpr int WN = (QB - 1) * SW + 3;
            const int wbase = q0 * SW - d.pw;
#pragma unroll
            for (int r = 0; r < 3; ++r) {
                const int h = p * d.sh - d.ph + r * d.dh;
                if (h < 0 || h >= d.H) continue;
                const T *xrow = x + (((int64_t)n * d.H + h) * d.W) * d.C + c0;
                uint4 win[WN];
#pragma unroll
                for (int t = 0; t < WN; ++t) {
                    const int ww = wbase + t;
                    win[t] = (ww >= 0 && ww < d.W) ? *reinterpret_cast<const uint4 *>(xrow + (int64_t)ww * d.C)
                                                    : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int s = 0; s < 3; ++s) {
                    const uint4 wq4 = *reinterpret_cast<const uint4 *>(w + (int64_t)(r * 3 + s) * d.C + c0);
                    const __half2 *wq = reinterpret_cast<const __half2 *>(&wq4);
#pragma unroll
                    for (int j = 0; j < QB; ++j) {
                        const __half2 *xv = reinterpret_cast<const __half2 *>(&win[j * SW + s]);
#pragma unroll
                        for (int k = 0; k < 4; ++k) hacc[j][k] = __hfma2(xv[k], wq[k], hacc[j][k]);
                    }
                }
            }
            T *yrow = y + ((int64_t)rowi * d.Q) * d.C + c0;
            const __half2 z2 = __float2half2_rn(0.0f), six2 = __float2half2_rn(6.0f);
#pragma unroll
            for (int j = 0; j < QB; ++j) {
                if (q0 + j >= d.Q) break;
                uint4 o;
                __half2 *oh = reinterpret_cast<__half2 *>(&o);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    __half2 v = hacc[j][k];
                    if (d.act == SN_ACT_RELU) {
                        v = __hmax2(v, z2);
                    } else if (d.act == SN_ACT_RELU6) {
                        v = __hmin2(__hmax2(v, z2), six2);
                    } else if (d.act != SN_ACT_NONE) {
                        const float2 f = __half22float2(v);
                        v = __floats2half2_rn(act_apply(f.x, d.act), act_apply(f.y, d.act));
                    }
                    oh[k] = v;
                }
                *reinterpret_cast<uint4 *>(yrow + (int64_t)(q0 + j) * d.C) = o;
            }
            continue;
        }
        float acc[QB][E];
#pragma unroll
        for (int j = 0; j < QB; ++j)
#pragma unroll
            for (int e = 0; e < E; ++e) acc[j][e] = b[e];
        if (SW > 0) {
            // 3x3 fast path: the input window of each tap row (QB outputs need
            // (QB-1)*SW + 3 columns) is loaded once and reused by the three taps
            constexpr int WN = (QB - 1) * (SW > 0 ? SW : 1) + 3;
            const int wbase = q0 * SW - d.pw;
#pragma unroll
            for (int r = 0; r < 3; ++r) {
                const int h = p * d.sh - d.ph + r * d.dh;
                if (h < 0 || h >= d.H) continue;
                const T *xrow = x + (((int64_t)n * d.H + h) * d.W) * d.C + c0;
                uint4 win[WN];
#pragma unroll
                for (int t = 0; t < WN; ++t) {
                    const int ww = wbase + t;
                    win[t] = (ww >= 0 && ww < d.W) ? *reinterpret_cast<const uint4 *>(xrow + (int64_t)ww * d.C)
                                                    : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int s = 0; s < 3; ++s) {
                    const uint4 wq = *reinterpret_cast<const uint4 *>(w + (int64_t)(r * 3 + s) * d.C + c0);
#pragma unroll
                    for (int j = 0; j < QB; ++j) fma16<T>(acc[j], win[j * (SW > 0 ? SW : 1) + s], wq);
                }
            }
        } else {
            for (int r = 0; r < d.R; ++r) {
                const int h = p * d.sh - d.ph + r * d.dh;
                if (h < 0 || h >= d.H) continue;
                const T *xrow = x + (((int64_t)n * d.H + h) * d.W) * d.C + c0;
                for (int s = 0; s < d.S; ++s) {
                    const uint4 wq = *reinterpret_cast<const uint4 *>(w + (int64_t)(r * d.S + s) * d.C + c0);
#pragma unroll
                    for (int j = 0; j < QB; ++j) {
                        const int ww = (q0 + j) * d.sw - d.pw + s * d.dw;
                        if (q0 + j < d.Q && ww >= 0 && ww < d.W)
                            fma16<T>(acc[j], *reinterpret_cast<const uint4 *>(xrow + (int64_t)ww * d.C), wq);
                    }
                }
            }
        }
        T *yrow = y + ((int64_t)rowi * d.Q) * d.C + c0;
#pragma unroll
        for (int j = 0; j < QB; ++j) {
            if (q0 + j >= d.Q) break;
            uint4 o;
            T *op = reinterpret_cast<T *>(&o);
#pragma unroll
            for (int e = 0; e < E; ++e) op[e] = cvt<T>(act_apply(acc[j][e], d.act));
            *reinterpret_cast<uint4 *>(yrow + (int64_t)(q0 + j) * d.C) = o;
        }
    }
}

// asynchronous 16-byte global -> shared copy, zero-filled when !valid
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem, bool valid) {
    const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(sa), "l"(gmem), "r"(valid ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// 3x3 depthwise, NHWC, small maps (stride 1 or 2, padding 1): one CTA per
// (image, 128-byte channel slice, band of PB output rows).  The band's input
// rows -- every column of the slice, with the zero padding around -- are read
// once, 16 bytes a thread and 128 bytes a pixel (coalesced), into shared
// memory; each thread then keeps one channel vector's nine tap weights in
// registers and produces that vector for output pixel after pixel from the
// shared tile, writing 16-byte vectors.  Input bytes cross HBM once (plus the
// two halo rows of a band), so the kernel needs no cross-thread reuse through
// L1 and no per-thread windows.  The accumulation order is that of the other
// NHWC kernels (bias, then rows inside the image, then columns), so the
// results agree with them bit for bit.
template <typename T, int SW>
__global__ void __launch_bounds__(256, 4) dw3_nhwc_band(const T *__restrict__ x, const T *__restrict__ w,
                                                     const float *__restrict__ bias, T *__restrict__ y, ConvDims d,
                                                     int PB) {
    griddep_launch();
    griddep_wait();
    constexpr int E = 16 / sizeof(T);  // elements per 16-byte vector
    constexpr int VS = 8;              // vectors per 128-byte slice
    extern __shared__ uint4 band_smem[];
    const int slices = (d.C * (int)sizeof(T) + 127) / 128;
    const int slice = (int)(blockIdx.x % slices), band = (int)(blockIdx.x / slices);
    const int n = blockIdx.y;
    const int p0 = band * PB, p1 = min(p0 + PB, d.P);
    const int h0 = p0 * SW - 1;              // input row of band row 0 (padding 1)
    const int rows = (p1 - p0 - 1) * SW + 3;
    const int WP = d.W + 2;                  // band columns, padding included
    const int nv = min(VS, (d.C * (int)sizeof(T) - slice * 128) / 16);  // vectors of this slice
    const int cs = slice * (128 / (int)sizeof(T));
    // asynchronous 16-byte copies (zero-filled outside the image and the
    // slice): every load of the band is in flight at once, none holds a
    // register
    for (int i = threadIdx.x; i < rows * WP * VS; i += blockDim.x) {
        const int v = i % VS, pix = i / VS, rr = pix / WP, cc = pix - rr * WP;
        const int h = h0 + rr, ww = cc - 1;
        const bool ok = v < nv && h >= 0 && h < d.H && ww >= 0 && ww < d.W;
        const T *src = ok ? x + (((int64_t)n * d.H + h) * d.W + ww) * d.C + cs + v * E : x;
        cp_async16(band_smem + i, src, ok);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    const int v = threadIdx.x % VS;
    if (v >= nv) return;  // no barrier follows
    const int c0 = cs + v * E;
    uint4 wv[9];
#pragma unroll
    for (int k = 0; k < 9; ++k) wv[k] = *reinterpret_cast<const uint4 *>(w + (int64_t)k * d.C + c0);
    float b[E];
#pragma unroll
    for (int e = 0; e < E; ++e) b[e] = bias[c0 + e];
    for (int o = threadIdx.x / VS; o < (p1 - p0) * d.Q; o += blockDim.x / VS) {
        const int pr = o / d.Q, q = o - pr * d.Q;
        const int hb = (p0 + pr) * SW - 1;  // input row of tap row 0
        uint4 out;
        if constexpr (std::is_same<T, __half>::value) {
            __half2 hacc[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) hacc[k] = __floats2half2_rn(b[2 * k], b[2 * k + 1]);
#pragma unroll
            for (int r = 0; r < 3; ++r) {
                if (hb + r < 0 || hb + r >= d.H) continue;
                const uint4 *row = band_smem + ((pr * SW + r) * WP + q * SW) * VS + v;
#pragma unroll
                for (int s_ = 0; s_ < 3; ++s_) {
                    const uint4 xv4 = row[s_ * VS];
                    const __half2 *xv = reinterpret_cast<const __half2 *>(&xv4);
                    const __half2 *wq = reinterpret_cast<const __half2 *>(&wv[r * 3 + s_]);
#pragma unroll
                    for (int k = 0; k < 4; ++k) hacc[k] = __hfma2(xv[k], wq[k], hacc[k]);
                }
            }
            __half2 *oh = reinterpret_cast<__half2 *>(&out);
            const __half2 z2 = __float2half2_rn(0.0f), six2 = __float2half2_rn(6.0f);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                __half2 vv = hacc[k];
                if (d.act == SN_ACT_RELU) {
                    vv = __hmax2(vv, z2);
                } else if (d.act == SN_ACT_RELU6) {
                    vv = __hmin2(__hmax2(vv, z2), six2);
                } else if (d.act != SN_ACT_NONE) {
                    const float2 f = __half22float2(vv);
                    vv = __floats2half2_rn(act_apply(f.x, d.act), act_apply(f.y, d.act));
                }
                oh[k] = vv;
            }
        } else {
            float acc[E];
#pragma unroll
            for (int e = 0; e < E; ++e) acc[e] = b[e];
#pragma unroll
            for (int r = 0; r < 3; ++r) {
                if (hb + r < 0 || hb + r >= d.H) continue;
                const uint4 *row = band_smem + ((pr * SW + r) * WP + q * SW) * VS + v;
#pragma unroll
                for (int s_ = 0; s_ < 3; ++s_) fma16<T>(acc, row[s_ * VS], wv[r * 3 + s_]);
            }
            T *op = reinterpret_cast<T *>(&out);
#pragma unroll
            for (int e = 0; e < E; ++e) op[e] = cvt<T>(act_apply(acc[e], d.act));
        }
        *reinterpret_cast<uint4 *>(y + (((int64_t)n * d.P + p0 + pr) * d.Q + q) * d.C + c0) = out;
    }
}

// band height and shared-memory bytes of dw3_nhwc_band for a layer (PB = 0:
// the kernel does not apply: a 3-row band of the map would not fit)
static int dw3_band_rows(const ConvDims &d, size_t *smem) {
    const size_t row_bytes = (size_t)(d.W + 2) * 128;
    const size_t budget = d.W <= 64 ? 32768 : 49152;
    const int max_rows = (int)(budget / row_bytes);
    if (max_rows < 3) return 0;
    int PB = (max_rows - 3) / d.sh + 1;
    if (PB > d.P) PB = d.P;
    *smem = (size_t)((PB - 1) * d.sh + 3) * row_bytes;
    return PB;
}

// NCHW: one thread per (n, c, p) and 8 consecutive output columns; consecutive
// threads take consecutive column blocks, so every load and store is
// coalesced across the warp; weights are [C][R][S].
template <typename T>
__global__ void __launch_bounds__(256) dw_nchw_row(const T *__restrict__ x, const T *__restrict__ w,
                                                   const float *__restrict__ bias, T *__restrict__ y, ConvDims d) {
    griddep_launch();
    griddep_wait();
    constexpr int QB = 8;
    const int QBLK = (d.Q + QB - 1) / QB;
    const int64_t total = (int64_t)d.N * d.C * d.P * QBLK;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int qb = (int)(i % QBLK);
        int64_t rest = i / QBLK;
        const int p = (int)(rest % d.P);
        const int64_t nc = rest / d.P;
        const int c = (int)(nc % d.C);
        const int q0 = qb * QB;
        const T *xc = x + nc * d.H * (int64_t)d.W;
        const T *wc = w + (int64_t)c * d.R * d.S;
        const float bv = bias[c];
        float acc[QB];
#pragma unroll
        for (int j = 0; j < QB; ++j) acc[j] = bv;
        for (int r = 0; r < d.R; ++r) {
            const int h = p * d.sh - d.ph + r * d.dh;
            if (h < 0 || h >= d.H) continue;
            const T *xr = xc + (int64_t)h * d.W;
            for (int s = 0; s < d.S; ++s) {
                const float wv = ldf<T>(wc + r * d.S + s);
#pragma unroll
                for (int j = 0; j < QB; ++j) {
                    const int ww = (q0 + j) * d.sw - d.pw + s * d.dw;
                    if (q0 + j < d.Q && ww >= 0 && ww < d.W) acc[j] = fmaf(ldf<T>(xr + ww), wv, acc[j]);
                }
            }
        }
        T *yr = y + (nc * d.P + p) * (int64_t)d.Q;
        if (sizeof(T) == 2 && q0 + QB <= d.Q && ((uintptr_t)(yr + q0) & 15) == 0) {
            uint4 o;
            T *op = reinterpret_cast<T *>(&o);
#pragma unroll
            for (int j = 0; j < QB; ++j) op[j] = cvt<T>(act_apply(acc[j], d.act));
            *reinterpret_cast<uint4 *>(yr + q0) = o;
        } else {
#pragma unroll
            for (int j = 0; j < QB; ++j)
                if (q0 + j < d.Q) stf<T>(yr + q0 + j, act_apply(acc[j], d.act));
        }
    }
}

// NHWC 3x3 (dilation 1) with shared-memory halo staging.  A work unit is TP
// x TQ output pixels of one image and a 128-byte slice of channels; its input
// halo ((TP-1)*SW+3 rows x (TQ-1)*SW+3 columns x 128 bytes) is copied into
// shared memory with cp.async (zero-filled outside the image, which is the
// padding).  The CTA is persistent with a ring of STAGES halo buffers: the
// halos of its next STAGES-1 units are in flight while the current one is
// computed from shared memory.
// Every input byte comes from DRAM once (plus the halo overlap) and the nine
// taps are served by shared memory.
constexpr int DW_TP = 8;
template <int SW> struct DwTQ { static constexpr int v = SW == 1 ? 16 : 8; };  // output columns per unit


template <typename T, int SW, int STAGES>
__global__ void __launch_bounds__(256, 2) dw3_nhwc_halo(const T *__restrict__ x, const T *__restrict__ w,
                                                        const float *__restrict__ bias, T *__restrict__ y, ConvDims d) {
    griddep_launch();
    griddep_wait();
    constexpr int DW_TQ = DwTQ<SW>::v;
    constexpr int E = 16 / sizeof(T);          // elements per 16-byte vector
    constexpr int VS = 8;                      // vectors per 128-byte channel slice
    constexpr int IH = (DW_TP - 1) * SW + 3, IW = (DW_TQ - 1) * SW + 3;
    constexpr int HALO = IH * IW * VS;         // 16-byte vectors per buffer
    extern __shared__ uint4 halo_smem[];
    const int slices = (d.C * (int)sizeof(T) + 127) / 128;
    const int tpn = (d.P + DW_TP - 1) / DW_TP, tqn = (d.Q + DW_TQ - 1) / DW_TQ;
    const int64_t units = (int64_t)d.N * tpn * tqn * slices;
    const int CV = d.C / E;  // 16-byte vectors per pixel
    auto issue = [&](int64_t u, uint4 *buf) {
        const int cs = (int)(u % slices);
        int64_t r = u / slices;
        const int tq = (int)(r % tqn);
        r /= tqn;
        const int tp = (int)(r % tpn);
        const int64_t n = r / tpn;
        const int h0 = tp * DW_TP * SW - d.ph, w0 = tq * DW_TQ * SW - d.pw;
        for (int i = threadIdx.x; i < HALO; i += blockDim.x) {
            const int v = i % VS, px = i / VS, ih = px / IW, iw = px % IW;
            const int h = h0 + ih, ww = w0 + iw, cv = cs * VS + v;
            const bool ok = h >= 0 && h < d.H && ww >= 0 && ww < d.W && cv < CV;
            const T *src = ok ? x + (((n * d.H + h) * d.W + ww) * (int64_t)d.C + (int64_t)cv * E) : x;
            cp_async16(buf + i, src, ok);
        }
        cp_async_commit();
    };
    const int v = threadIdx.x % VS;  // this thread's vector within the slice
    // prologue: the first STAGES-1 units of this CTA in flight
    for (int k = 0; k < STAGES - 1; ++k) {
        const int64_t uk = blockIdx.x + (int64_t)k * gridDim.x;
        if (uk < units) issue(uk, halo_smem + k * HALO);
        else cp_async_commit();  // keep the group count uniform
    }
    int buf = 0;
    for (int64_t u = blockIdx.x; u < units; u += gridDim.x, buf = (buf + 1) % STAGES) {
        const int64_t un = u + (int64_t)(STAGES - 1) * gridDim.x;
        if (un < units) issue(un, halo_smem + ((buf + STAGES - 1) % STAGES) * HALO);
        else cp_async_commit();
        cp_async_wait<STAGES - 1>();  // the current unit's halo has landed
        __syncthreads();
        const uint4 *hb = halo_smem + buf * HALO;
        const int cs = (int)(u % slices);
        int64_t r = u / slices;
        const int tq = (int)(r % tqn);
        r /= tqn;
        const int tp = (int)(r % tpn);
        const int64_t n = r / tpn;
        const int cv = cs * VS + v;
        if (cv < CV) {
            const int c0 = cv * E;
            float wf[9][E], bv[E];
#pragma unroll
            for (int t = 0; t < 9; ++t) {
                const uint4 wq = *reinterpret_cast<const uint4 *>(w + (int64_t)t * d.C + c0);
                const T *wp = reinterpret_cast<const T *>(&wq);
#pragma unroll
                for (int e = 0; e < E; ++e) wf[t][e] = ldf<T>(wp + e);
            }
#pragma unroll
            for (int e = 0; e < E; ++e) bv[e] = bias[c0 + e];
            for (int px = threadIdx.x / VS; px < DW_TP * DW_TQ; px += blockDim.x / VS) {
                const int op = px / DW_TQ, oq = px % DW_TQ;
                const int p = tp * DW_TP + op, q = tq * DW_TQ + oq;
                if (p >= d.P || q >= d.Q) continue;
                float acc[E];
#pragma unroll
                for (int e = 0; e < E; ++e) acc[e] = bv[e];
#pragma unroll
                for (int rr = 0; rr < 3; ++rr)
#pragma unroll
                    for (int ss = 0; ss < 3; ++ss) {
                        const uint4 xq = hb[((op * SW + rr) * IW + oq * SW + ss) * VS + v];
                        const T *xp = reinterpret_cast<const T *>(&xq);
#pragma unroll
                        for (int e = 0; e < E; ++e) acc[e] = fmaf(ldf<T>(xp + e), wf[rr * 3 + ss][e], acc[e]);
                    }
                uint4 o;
                T *opp = reinterpret_cast<T *>(&o);
#pragma unroll
                for (int e = 0; e < E; ++e) opp[e] = cvt<T>(act_apply(acc[e], d.act));
                *reinterpret_cast<uint4 *>(y + ((n * d.P + p) * (int64_t)d.Q + q) * d.C + c0) = o;
            }
        }
        __syncthreads();  // everyone is done with this buffer before it is refilled
    }
}

// NCHW 3x3: a block owns TH output rows of one (n, c) plane.  The input rows
// they need (contiguous in NCHW) are staged in shared memory with coalesced
// loads, zero-padded left/right and outside the image; then consecutive
// threads compute consecutive outputs of the tile, so the stores are
// coalesced too.  Weights are [C][3][3].
template <typename T>
__global__ void __launch_bounds__(256) dw3_nchw_tile(const T *__restrict__ x, const T *__restrict__ w,
                                                     const float *__restrict__ bias, T *__restrict__ y, ConvDims d,
                                                     int TH) {
    griddep_launch();
    griddep_wait();
    extern __shared__ float dw_tile[];
    const int tiles = (d.P + TH - 1) / TH;
    const int64_t nc = blockIdx.x / tiles;
    const int p0 = (int)(blockIdx.x % tiles) * TH;
    const int c = (int)(nc % d.C);
    const int rows = (TH - 1) * d.sh + 1 + 2 * d.dh;  // input rows touched by TH output rows
    const int WP = d.W + 2 * d.pw;                     // padded width
    const int h0 = p0 * d.sh - d.ph;
    const T *xc = x + nc * d.H * (int64_t)d.W;
    for (int i = threadIdx.x; i < rows * WP; i += blockDim.x) {
        const int rr = i / WP, cc = i - rr * WP;
        const int h = h0 + rr, ww = cc - d.pw;
        dw_tile[i] = (h >= 0 && h < d.H && ww >= 0 && ww < d.W) ? ldf<T>(xc + (int64_t)h * d.W + ww) : 0.f;
    }
    float wr[9];
#pragma unroll
    for (int t = 0; t < 9; ++t) wr[t] = ldf<T>(w + (int64_t)c * 9 + t);
    const float bv = bias[c];
    __syncthreads();
    const int pend = min(TH, d.P - p0);
    T *yc = y + nc * d.P * (int64_t)d.Q;
    for (int i = threadIdx.x; i < pend * d.Q; i += blockDim.x) {
        const int pr = i / d.Q, q = i - pr * d.Q;
        const float *base = dw_tile + (pr * d.sh) * WP + q * d.sw;
        float acc = bv;
#pragma unroll
        for (int r = 0; r < 3; ++r)
#pragma unroll
            for (int s = 0; s < 3; ++s) acc = fmaf(base[r * d.dh * WP + s * d.dw], wr[r * 3 + s], acc);
        stf<T>(yc + (int64_t)(p0 + pr) * d.Q + q, act_apply(acc, d.act));
    }
}

bool dw3_band_applies(const Layer &l, const Shape &in, sn_schema s) {
    const sn_conv_params &c = l.conv;
    if (s.dtype == SN_QI8 || s.layout != SN_NHWC || c.kh != 3 || c.kw != 3 || c.dh != 1 || c.dw != 1 ||
        c.ph != 1 || c.pw != 1 || c.sh != c.sw || (c.sh != 1 && c.sh != 2) || (in.c * dtype_size(s.dtype)) % 16 ||
        in.n > 65535)
        return false;
    const ConvDims d{(int32_t)in.n, (int32_t)in.c, (int32_t)in.h, (int32_t)in.w, c.c_out, (int32_t)l.out.h,
                     (int32_t)l.out.w, 3, 3, c.sh, c.sw, 1, 1, 1, 1, c.groups, c.act};
    size_t smem = 0;
    return dw3_band_rows(d, &smem) > 0;
}

cudaError_t dwconv(const LaunchArgs &a) {
    // routine parameter (variant): NHWC 0 = register window (4 columns per
    // thread), 1 = input rows staged by TMA in a shared-memory ring (3x3,
    // 16-bit; shared-memory halo tiles otherwise); NCHW 0 = row kernel (8
    // columns per thread), 1 = shared-memory plane tile
    const ConvDims d = conv_dims(a);
    if (a.variant == 1 && dw3_ring_applies(a, d)) {
        const cudaError_t e = dw3_nhwc_ring(a, d);
        if (e != cudaErrorNotSupported) return e;  // else the shared-memory halo kernel below
    }
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    const int es = dtype_size(a.schema.dtype);
    const bool vec_ok = (d.C * es) % 16 == 0 && (uintptr_t)a.in[0] % 16 == 0 && (uintptr_t)a.out % 16 == 0 &&
                        (uintptr_t)a.wt % 16 == 0;
    const bool k3 = d.R == 3 && d.S == 3 && d.dw == 1;
    SN_DT_SWITCH(a.schema.dtype, T, {
        const T *x = (const T *)a.in[0];
        const T *w = (const T *)a.wt;
        T *y = (T *)a.out;
        const bool band_ok = k3 && d.dh == 1 && d.ph == 1 && d.pw == 1 && d.sh == d.sw && (d.sh == 1 || d.sh == 2);
        size_t band_smem = 0;
        const int PB = band_ok && a.schema.layout == SN_NHWC && vec_ok ? dw3_band_rows(d, &band_smem) : 0;
        if (a.variant == 2 && PB > 0 && d.N <= 65535) {
            const int slices = (int)((d.C * (int64_t)es + 127) / 128);
            const dim3 gb((unsigned)(slices * ((d.P + PB - 1) / PB)), (unsigned)d.N);
            static bool attr = false;
            if (!attr) {
                cudaFuncSetAttribute(dw3_nhwc_band<T, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, 49152);
                cudaFuncSetAttribute(dw3_nhwc_band<T, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 49152);
                attr = true;
            }
            if (d.sh == 1) launch_pdl(dw3_nhwc_band<T, 1>, gb, 256, band_smem, a.stream, x, w, a.bias, y, d, PB);
            else launch_pdl(dw3_nhwc_band<T, 2>, gb, 256, band_smem, a.stream, x, w, a.bias, y, d, PB);
        } else if (a.schema.layout == SN_NHWC && vec_ok) {
            const int64_t cvec = d.C * es / 16;
            const bool halo = k3 && d.dh == 1 && (d.sw == 1 || d.sw == 2) && d.sh == d.sw;
            if (a.variant == 1 && halo) {
                const int slices = (int)((d.C * (int64_t)es + 127) / 128);
                const int tq = d.sw == 1 ? DwTQ<1>::v : DwTQ<2>::v;
                const int64_t units = (int64_t)d.N * ((d.P + DW_TP - 1) / DW_TP) * ((d.Q + tq - 1) / tq) * slices;
                const unsigned gb = (unsigned)std::min<int64_t>(units, 152LL * 2);
                static bool attr = false;
                const size_t sm1 = 4 * (size_t)((DW_TP - 1) + 3) * ((DwTQ<1>::v - 1) + 3) * 8 * 16;
                const size_t sm2 = 3 * (size_t)((DW_TP - 1) * 2 + 3) * ((DwTQ<2>::v - 1) * 2 + 3) * 8 * 16;
                if (!attr) {
                    cudaFuncSetAttribute(dw3_nhwc_halo<T, 1, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm1);
                    cudaFuncSetAttribute(dw3_nhwc_halo<T, 2, 3>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm2);
                    attr = true;
                }
                if (d.sw == 1) launch_pdl(dw3_nhwc_halo<T, 1, 4>, gb, 256, sm1, a.stream, x, w, a.bias, y, d);
                else launch_pdl(dw3_nhwc_halo<T, 2, 3>, gb, 256, sm2, a.stream, x, w, a.bias, y, d);
            } else {
                const int QBLK = (d.Q + 3) / 4, CV = (int)cvec;
                const dim3 gb((unsigned)((QBLK * CV + 255) / 256), (unsigned)std::min<int64_t>((int64_t)d.N * d.P, 65535));
                if (k3 && d.sw == 1) launch_pdl(dw_nhwc_vec<T, 4, 1>, gb, 256, 0, a.stream, x, w, a.bias, y, d, CV, QBLK);
                else if (k3 && d.sw == 2) launch_pdl(dw_nhwc_vec<T, 4, 2>, gb, 256, 0, a.stream, x, w, a.bias, y, d, CV, QBLK);
                else launch_pdl(dw_nhwc_vec<T, 4, 0>, gb, 256, 0, a.stream, x, w, a.bias, y, d, CV, QBLK);
            }
        } else if (a.schema.layout == SN_NHWC) {
            launch_pdl(dw_nhwc<T>, grid_for(total, 256), 256, 0, a.stream, x, w, a.bias, y, d);
        } else {
            bool tiled = false;
            if (a.variant == 1 && d.R == 3 && d.S == 3) {
                int TH = (int)std::max<int64_t>(1, std::min<int64_t>(d.P, 512 / std::max(1, d.Q)));
                auto tile_bytes = [&](int th) {
                    return (size_t)((th - 1) * d.sh + 1 + 2 * d.dh) * (d.W + 2 * d.pw) * sizeof(float);
                };
                while (tile_bytes(TH) > 40 * 1024 && TH > 1) TH /= 2;
                const int64_t blocks = (int64_t)d.N * d.C * ((d.P + TH - 1) / TH);
                if (tile_bytes(TH) <= 40 * 1024 && blocks < ((int64_t)1 << 31)) {
                    launch_pdl(dw3_nchw_tile<T>, (unsigned)blocks, 256, tile_bytes(TH), a.stream, x, w, a.bias, y, d, TH);
                    tiled = true;
                }
            }
            if (!tiled)
                launch_pdl(dw_nchw_row<T>, grid_for((int64_t)d.N * d.C * d.P * ((d.Q + 7) / 8), 256, 152LL * 16), 256, 0, a.stream, x, w, a.bias, y, d);
        }
    });
    return cudaGetLastError();
}

// ===========================================================================
// max pooling (-inf padding), global average pooling, add, dense
// ===========================================================================
template <typename T, bool NHWC>
__global__ void maxpool_kernel(const T *__restrict__ x, T *__restrict__ y, int N, int C, int H, int W,
                               int P, int Q, int kh, int kw, int sh, int sw, int ph, int pw) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)N * C * P * Q;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int c, p, q;
        int64_t n;
        if (NHWC) {
            c = (int)(i % C);
            const int64_t pix = i / C;
            q = (int)(pix % Q);
            p = (int)((pix / Q) % P);
            n = pix / ((int64_t)Q * P);
        } else {
            q = (int)(i % Q);
            p = (int)((i / Q) % P);
            c = (int)((i / ((int64_t)Q * P)) % C);
            n = i / ((int64_t)Q * P * C);
        }
        float m = -INFINITY;
        for (int r = 0; r < kh; ++r) {
            const int h = p * sh - ph + r;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < kw; ++s) {
                const int ww = q * sw - pw + s;
                if (ww < 0 || ww >= W) continue;
                const int64_t idx = NHWC ? ((n * H + h) * W + ww) * C + c : ((n * C + c) * H + h) * (int64_t)W + ww;
                m = fmaxf(m, ldf<T>(x + idx));
            }
        }
        stf<T>(y + i, m);
    }
}

// NHWC, 16 bytes of channels per thread (8 x 16-bit or 4 x fp32 lanes)
// NHWC, 16-byte channel vectors: the grid's y axis walks the N x P output
// rows, its x axis the (column, channel vector) pairs of a row, channel vector
// fastest (coalesced); 32-bit index math, one division per thread.  Packed
// 16-bit max (exact: the result is one of the stored values).
template <typename T>
__device__ __forceinline__ uint32_t max2(uint32_t a, uint32_t b);
template <>
__device__ __forceinline__ uint32_t max2<__half>(uint32_t a, uint32_t b) {
    const __half2 r = __hmax2(*reinterpret_cast<const __half2 *>(&a), *reinterpret_cast<const __half2 *>(&b));
    return *reinterpret_cast<const uint32_t *>(&r);
}
template <>
__device__ __forceinline__ uint32_t max2<__nv_bfloat16>(uint32_t a, uint32_t b) {
    const __nv_bfloat162 r =
        __hmax2(*reinterpret_cast<const __nv_bfloat162 *>(&a), *reinterpret_cast<const __nv_bfloat162 *>(&b));
    return *reinterpret_cast<const uint32_t *>(&r);
}
template <>
__device__ __forceinline__ uint32_t max2<float>(uint32_t a, uint32_t b) {
    return __float_as_uint(fmaxf(__uint_as_float(a), __uint_as_float(b)));
}

template <typename T>
__global__ void __launch_bounds__(256) maxpool_nhwc_vec(const uint4 *__restrict__ x, uint4 *__restrict__ y, int N,
                                                       int C16, int H, int W, int P, int Q, int kh, int kw, int sh,
                                                       int sw, int ph, int pw) {
    griddep_launch();
    griddep_wait();
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= Q * C16) return;
    const int q = t / C16, cv = t - q * C16;
    // -inf in every lane (16-bit: 0xfc00 half, 0xff80 bfloat16; fp32: 0xff800000)
    const uint32_t ninf = sizeof(T) == 4 ? 0xff800000u : (std::is_same<T, __half>::value ? 0xfc00fc00u : 0xff80ff80u);
    for (int row = blockIdx.y; row < N * P; row += gridDim.y) {
        const int n = row / P, p = row - n * P;
        uint4 m = make_uint4(ninf, ninf, ninf, ninf);
        for (int r = 0; r < kh; ++r) {
            const int h = p * sh - ph + r;
            if (h < 0 || h >= H) continue;
            const uint4 *xr = x + ((size_t)(n * H + h) * W) * C16 + cv;
            for (int s2 = 0; s2 < kw; ++s2) {
                const int ww = q * sw - pw + s2;
                if (ww < 0 || ww >= W) continue;
                const uint4 v = xr[(size_t)ww * C16];
                m.x = max2<T>(m.x, v.x);
                m.y = max2<T>(m.y, v.y);
                m.z = max2<T>(m.z, v.z);
                m.w = max2<T>(m.w, v.w);
            }
        }
        y[((size_t)row * Q + q) * C16 + cv] = m;
    }
}

cudaError_t maxpool(const LaunchArgs &a) {
    const Shape &i = a.in_shapes[0], &o = a.layer->out;
    const sn_pool_params &p = a.layer->pool;
    const int64_t total = o.numel();
    SN_DT_SWITCH(a.schema.dtype, T, {
        const int64_t cb = i.c * (int64_t)sizeof(T);
        if (a.schema.layout == SN_NHWC && cb % 16 == 0 && (uintptr_t)a.in[0] % 16 == 0 &&
            (uintptr_t)a.out % 16 == 0) {
            const int c16 = (int)(cb / 16);
            const dim3 g((unsigned)((o.w * c16 + 255) / 256), (unsigned)std::min<int64_t>(o.n * o.h, 65535));
            launch_pdl(maxpool_nhwc_vec<T>, g, 256, 0, a.stream, (const uint4 *)a.in[0], (uint4 *)a.out, (int)i.n,
                       c16, (int)i.h, (int)i.w, (int)o.h, (int)o.w, p.kh, p.kw, p.sh, p.sw, p.ph, p.pw);
        } else if (a.schema.layout == SN_NHWC)
            launch_pdl(maxpool_kernel<T, true>, grid_for(total, 256), 256, 0, a.stream, 
                (const T *)a.in[0], (T *)a.out, (int)i.n, (int)i.c, (int)i.h, (int)i.w, (int)o.h, (int)o.w,
                p.kh, p.kw, p.sh, p.sw, p.ph, p.pw);
        else
            launch_pdl(maxpool_kernel<T, false>, grid_for(total, 256), 256, 0, a.stream, 
                (const T *)a.in[0], (T *)a.out, (int)i.n, (int)i.c, (int)i.h, (int)i.w, (int)o.h, (int)o.w,
                p.kh, p.kw, p.sh, p.sw, p.ph, p.pw);
    });
    return cudaGetLastError();
}

// NCHW: one warp per (n, c) sums HW contiguous values
template <typename T>
__global__ void gap_nchw(const T *__restrict__ x, T *__restrict__ y, int64_t NC, int64_t HW) {
    griddep_launch();
    griddep_wait();
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / 32;
    const int lane = threadIdx.x % 32;
    for (int64_t nc = warp; nc < NC; nc += (int64_t)gridDim.x * blockDim.x / 32) {
        float s = 0.f;
        for (int64_t i = lane; i < HW; i += 32) s += ldf<T>(x + nc * HW + i);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) stf<T>(y + nc, s / (float)HW);
    }
}

// NHWC, 16-byte channel vectors: a block of 32 channel vectors x 8 pixel
// slices per (image, 32-vector group); each thread sums its slice's pixels in
// f32, the block adds the 8 slices in order through shared memory
template <typename T>
__global__ void __launch_bounds__(256) gap_nhwc_vec(const T *__restrict__ x, T *__restrict__ y, int C, int HW) {
    griddep_launch();
    griddep_wait();
    constexpr int E = 16 / sizeof(T);
    __shared__ float part[8][32][E + 1];
    const int cvl = threadIdx.x & 31, sl = threadIdx.x >> 5;
    const int n = blockIdx.y;
    const int CV = C / E;
    const int cv = blockIdx.x * 32 + cvl;
    float s[E];
#pragma unroll
    for (int e = 0; e < E; ++e) s[e] = 0.f;
    if (cv < CV) {
        const T *xn = x + (size_t)n * HW * C + (size_t)cv * E;
        for (int p = sl; p < HW; p += 8) {
            const uint4 v = *reinterpret_cast<const uint4 *>(xn + (size_t)p * C);
            const T *pv = reinterpret_cast<const T *>(&v);
#pragma unroll
            for (int e = 0; e < E; ++e) s[e] += ldf<T>(pv + e);
        }
    }
#pragma unroll
    for (int e = 0; e < E; ++e) part[sl][cvl][e] = s[e];
    __syncthreads();
    if (sl == 0 && cv < CV) {
        uint4 o;
        T *po = reinterpret_cast<T *>(&o);
#pragma unroll
        for (int e = 0; e < E; ++e) {
            float t = 0.f;
            for (int k = 0; k < 8; ++k) t += part[k][cvl][e];
            po[e] = cvt<T>(t / (float)HW);
        }
        *reinterpret_cast<uint4 *>(y + (size_t)n * C + (size_t)cv * E) = o;
    }
}

// NHWC: one thread per (n, c); consecutive threads read consecutive channels
template <typename T>
__global__ void gap_nhwc(const T *__restrict__ x, T *__restrict__ y, int64_t N, int64_t C, int64_t HW) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < N * C;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t n = i / C, c = i % C;
        float s = 0.f;
        for (int64_t p = 0; p < HW; ++p) s += ldf<T>(x + (n * HW + p) * C + c);
        stf<T>(y + i, s / (float)HW);
    }
}

cudaError_t gap(const LaunchArgs &a) {
    const Shape &i = a.in_shapes[0];
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (a.schema.layout == SN_NCHW)
            launch_pdl(gap_nchw<T>, grid_for(i.n * i.c * 32, 256), 256, 0, a.stream, (const T *)a.in[0], (T *)a.out,
                                                                               i.n * i.c, i.h * i.w);
        else if ((i.c * (int64_t)sizeof(T)) % 16 == 0 && (uintptr_t)a.in[0] % 16 == 0 && (uintptr_t)a.out % 16 == 0 &&
                 i.n <= 65535 && i.h * i.w * i.c < ((int64_t)1 << 31)) {
            const int CV = (int)(i.c * (int64_t)sizeof(T) / 16);
            launch_pdl(gap_nhwc_vec<T>, dim3((unsigned)((CV + 31) / 32), (unsigned)i.n), 256, 0, a.stream,
                       (const T *)a.in[0], (T *)a.out, (int)i.c, (int)(i.h * i.w));
        } else
            launch_pdl(gap_nhwc<T>, grid_for(i.n * i.c, 256), 256, 0, a.stream, (const T *)a.in[0], (T *)a.out, i.n,
                                                                         i.c, i.h * i.w);
    });
    return cudaGetLastError();
}

template <typename T>
__global__ void add_kernel(const T *__restrict__ a, const T *__restrict__ b, T *__restrict__ y, int64_t n,
                           int act) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        stf<T>(y + i, act_apply(ldf<T>(a + i) + ldf<T>(b + i), act));
}

// 8 x 16-bit lanes per thread when everything is 16-byte aligned
template <typename T>
__global__ void add16_kernel(const uint4 *__restrict__ a, const uint4 *__restrict__ b, uint4 *__restrict__ y,
                             int64_t n16, int act) {
    griddep_launch();
    griddep_wait();
    constexpr int E = 16 / sizeof(T);
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint4 va = a[i], vb = b[i];
        uint4 vo;
        const T *pa = reinterpret_cast<const T *>(&va), *pb = reinterpret_cast<const T *>(&vb);
        T *po = reinterpret_cast<T *>(&vo);
#pragma unroll
        for (int e = 0; e < E; ++e) po[e] = cvt<T>(act_apply(ldf<T>(pa + e) + ldf<T>(pb + e), act));
        y[i] = vo;
    }
}

cudaError_t add(const LaunchArgs &a) {
    const int64_t n = a.layer->out.numel();
    SN_DT_SWITCH(a.schema.dtype, T, {
        const int64_t bytes = n * (int64_t)sizeof(T);
        if (bytes % 16 == 0 && (uintptr_t)a.in[0] % 16 == 0 && (uintptr_t)a.in[1] % 16 == 0 &&
            (uintptr_t)a.out % 16 == 0)
            launch_pdl(add16_kernel<T>, grid_for(bytes / 16, 256), 256, 0, a.stream, 
                (const uint4 *)a.in[0], (const uint4 *)a.in[1], (uint4 *)a.out, bytes / 16, a.layer->act);
        else
            launch_pdl(add_kernel<T>, grid_for(n, 256), 256, 0, a.stream, (const T *)a.in[0], (const T *)a.in[1],
                                                                   (T *)a.out, n, a.layer->act);
    });
    return cudaGetLastError();
}

// per-channel scale: y[n,c,h,w] = act(x[n,c,h,w] * s[n,c]).  NHWC, 16-byte
// vectors when C allows: one thread per 8 (16-bit) or 4 (fp32) channels of a
// pixel; otherwise one thread per element, (n, c) from the layout.
template <typename T>
__global__ void mul_nhwc_vec(const uint4 *__restrict__ x, const T *__restrict__ s, uint4 *__restrict__ y,
                             int64_t pixels, int64_t HW, int CV, int act) {
    griddep_launch();
    griddep_wait();
    constexpr int E = 16 / sizeof(T);
    const int64_t total = pixels * CV;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t pix = i / CV;
        const int cv = (int)(i - pix * CV);
        const int64_t n = pix / HW;
        const uint4 xv = x[i];
        const uint4 sv = reinterpret_cast<const uint4 *>(s + n * (int64_t)CV * E)[cv];
        uint4 o;
        const T *px = reinterpret_cast<const T *>(&xv), *ps = reinterpret_cast<const T *>(&sv);
        T *po = reinterpret_cast<T *>(&o);
#pragma unroll
        for (int e = 0; e < E; ++e) po[e] = cvt<T>(act_apply(ldf<T>(px + e) * ldf<T>(ps + e), act));
        y[i] = o;
    }
}

template <typename T, bool NHWC>
__global__ void mul_kernel(const T *__restrict__ x, const T *__restrict__ s, T *__restrict__ y, int64_t n,
                           int64_t C, int64_t HW, int act) {
    griddep_launch();
    griddep_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t nc = NHWC ? (i / (HW * C)) * C + i % C : i / HW;  // index of (n, c) in s
        stf<T>(y + i, act_apply(ldf<T>(x + i) * ldf<T>(s + nc), act));
    }
}

cudaError_t mul(const LaunchArgs &a) {
    const Shape &o = a.layer->out;
    const int64_t n = o.numel(), HW = o.h * o.w;
    SN_DT_SWITCH(a.schema.dtype, T, {
        const int64_t cb = o.c * (int64_t)sizeof(T);
        if (a.schema.layout == SN_NHWC && cb % 16 == 0 && (uintptr_t)a.in[0] % 16 == 0 &&
            (uintptr_t)a.in[1] % 16 == 0 && (uintptr_t)a.out % 16 == 0)
            launch_pdl(mul_nhwc_vec<T>, grid_for(n * (int64_t)sizeof(T) / 16, 256), 256, 0, a.stream,
                       (const uint4 *)a.in[0], (const T *)a.in[1], (uint4 *)a.out, o.n * HW, HW, (int)(cb / 16),
                       a.layer->act);
        else if (a.schema.layout == SN_NHWC)
            launch_pdl(mul_kernel<T, true>, grid_for(n, 256), 256, 0, a.stream, (const T *)a.in[0],
                       (const T *)a.in[1], (T *)a.out, n, o.c, HW, a.layer->act);
        else
            launch_pdl(mul_kernel<T, false>, grid_for(n, 256), 256, 0, a.stream, (const T *)a.in[0],
                       (const T *)a.in[1], (T *)a.out, n, o.c, HW, a.layer->act);
    });
    return cudaGetLastError();
}

// dense: one warp per (n, o), dot product over the input features
template <typename T>
__global__ void dense_kernel(const T *__restrict__ x, const T *__restrict__ w, const float *__restrict__ bias,
                             T *__restrict__ y, int64_t N, int64_t IN, int64_t OUT, int act) {
    griddep_launch();
    griddep_wait();
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / 32;
    const int lane = threadIdx.x % 32;
    for (int64_t no = warp; no < N * OUT; no += (int64_t)gridDim.x * blockDim.x / 32) {
        const int64_t n = no / OUT, o = no % OUT;
        float s = 0.f;
        for (int64_t i = lane; i < IN; i += 32) s += ldf<T>(x + n * IN + i) * ldf<T>(w + o * IN + i);
        for (int k = 16; k > 0; k >>= 1) s += __shfl_xor_sync(0xffffffffu, s, k);
        if (lane == 0) stf<T>(y + no, act_apply(s + bias[o], act));
    }
}

cudaError_t dense(const LaunchArgs &a) {
    const Shape &i = a.in_shapes[0];
    const int64_t N = i.n, IN = a.layer->dense_in, OUT = a.layer->dense_out;
    SN_DT_SWITCH(a.schema.dtype, T,
                 launch_pdl(dense_kernel<T>, grid_for(N * OUT * 32, 256), 256, 0, a.stream, 
                     (const T *)a.in[0], (const T *)a.wt, a.bias, (T *)a.out, N, IN, OUT, a.layer->act));
    return cudaGetLastError();
}

}  // namespace k
}  // namespace sn
