// Adapt conversion, weight formatting, direct convolution, depthwise
// convolution, pooling, elementwise add and dense routines (CUDA cores).
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
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        stf<To>(y + i, ldf<Ti>(x + i));
}

// 16-byte vectorised copy when dtypes match
__global__ void copy16_kernel(const uint4 *__restrict__ x, uint4 *__restrict__ y, int64_t n16) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16;
         i += (int64_t)gridDim.x * blockDim.x)
        y[i] = x[i];
}

// batched transpose y[b][c][r] = x[b][r][c] with a cast, through a 64x64
// shared-memory tile (256 threads, 16 elements each); rows of 64 contiguous
// elements are read and written by consecutive threads.
constexpr int TT = 64;
template <typename Ti, typename To>
__global__ void __launch_bounds__(256) transpose_kernel(const Ti *__restrict__ x, To *__restrict__ y,
                                                         int64_t R, int64_t Cc) {
    __shared__ float tile[TT][TT + 1];
    const int64_t b = blockIdx.z;
    const int64_t r0 = (int64_t)blockIdx.y * TT, c0 = (int64_t)blockIdx.x * TT;
    const Ti *xb = x + b * R * Cc;
    To *yb = y + b * R * Cc;
    const int tx = threadIdx.x % TT, ty = threadIdx.x / TT;  // 64 x 4
#pragma unroll
    for (int i = 0; i < TT; i += 4) {
        const int64_t r = r0 + ty + i, c = c0 + tx;
        if (r < R && c < Cc) tile[ty + i][tx] = ldf<Ti>(xb + r * Cc + c);
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < TT; i += 4) {
        const int64_t c = c0 + ty + i, r = r0 + tx;
        if (r < R && c < Cc) stf<To>(yb + c * R + r, tile[tx][ty + i]);
    }
}

// few channels (C <= 16): one thread per pixel moves all of its channels;
// the planar side is read/written coalesced across threads, the interleaved
// side as C consecutive elements per thread (C * 32 contiguous per warp)
template <typename Ti, typename To, bool TO_NHWC>
__global__ void permute_small_c_kernel(const Ti *__restrict__ x, To *__restrict__ y, int64_t N, int C, int64_t HW) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < N * HW;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t n = i / HW, hw = i % HW;
        for (int c = 0; c < C; ++c) {
            const int64_t planar = (n * C + c) * HW + hw, inter = i * C + c;
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
                copy16_kernel<<<grid_for(bytes / 16, 256), 256, 0, st>>>((const uint4 *)x, (uint4 *)y,
                                                                          bytes / 16);
                return cudaGetLastError();
            }
            return cudaMemcpyAsync(y, x, bytes, cudaMemcpyDeviceToDevice, st);
        }
        cast_kernel<Ti, To><<<grid_for(n, 256), 256, 0, st>>>((const Ti *)x, (To *)y, n);
        return cudaGetLastError();
    }
    if (s.c <= 16) {
        const int64_t px = s.n * s.h * s.w;
        if (lay_in == SN_NCHW)
            permute_small_c_kernel<Ti, To, true><<<grid_for(px, 256), 256, 0, st>>>((const Ti *)x, (To *)y, s.n,
                                                                                     (int)s.c, s.h * s.w);
        else
            permute_small_c_kernel<Ti, To, false><<<grid_for(px, 256), 256, 0, st>>>((const Ti *)x, (To *)y, s.n,
                                                                                      (int)s.c, s.h * s.w);
        return cudaGetLastError();
    }
    // NCHW -> NHWC: per image [C][HW] -> [HW][C]; NHWC -> NCHW: [HW][C] -> [C][HW]
    const int64_t R = (lay_in == SN_NCHW) ? s.c : s.h * s.w;
    const int64_t Cc = (lay_in == SN_NCHW) ? s.h * s.w : s.c;
    if (s.n > 65535) return cudaErrorInvalidValue;
    dim3 grid((unsigned)((Cc + TT - 1) / TT), (unsigned)((R + TT - 1) / TT), (unsigned)s.n);
    if (grid.y > 65535) return cudaErrorInvalidValue;
    transpose_kernel<Ti, To><<<grid, 256, 0, st>>>((const Ti *)x, (To *)y, R, Cc);
    return cudaGetLastError();
}

cudaError_t convert(const void *x, int dt_in, int lay_in, void *y, int dt_out, int lay_out, Shape s,
                    cudaStream_t st) {
    SN_DT_SWITCH(dt_in, Ti, SN_DT_SWITCH(dt_out, To, return convert_t<Ti, To>(x, lay_in, y, lay_out, s, st)));
    return cudaErrorInvalidValue;
}

// deterministic pseudo-random fill in [-scale, scale)
template <typename T>
__global__ void fill_kernel(T *y, int64_t n, uint32_t seed, float scale) {
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
    SN_DT_SWITCH(dt, T, fill_kernel<T><<<grid_for(n, 256), 256, 0, st>>>((T *)y, n, seed, scale));
    return cudaGetLastError();
}

// ===========================================================================
// weight formats (from fp32 [K][Cg][R][S])
// ===========================================================================
template <typename T>
__global__ void weight_perm_kernel(const float *__restrict__ w, T *__restrict__ out, int fmt,
                                   int64_t K, int64_t Cg, int64_t R, int64_t S) {
    const int64_t total = K * Cg * R * S;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        // i indexes the source [k][c][r][s]
        const int64_t s = i % S, r = (i / S) % R, c = (i / (S * R)) % Cg, kk = i / (S * R * Cg);
        int64_t o;
        if (fmt == W_KCRS) o = i;
        else if (fmt == W_RSCK) o = ((r * S + s) * Cg + c) * K + kk;
        else if (fmt == W_KRSC_PAD64) o = kk * ((Cg * R * S + 63) / 64 * 64) + (r * S + s) * Cg + c;
        else o = ((kk * R + r) * S + s) * Cg + c;  // W_KRSC
        stf<T>(out + o, w[i]);
    }
}

// Winograd F(2x2,3x3) filter transform U = G g G^T (Lavin & Gray), stored
// [16][K][C] so that every xi = 4*a + b is a K x C row-major matrix.
template <typename T>
__global__ void weight_wino_kernel(const float *__restrict__ w, T *__restrict__ out, int64_t K,
                                   int64_t C) {
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

cudaError_t weight_format(const float *w, void *out, int fmt, int dt, int64_t K, int64_t Cg,
                          int64_t R, int64_t S, cudaStream_t st) {
    if (fmt == W_WINO) {
        if (R != 3 || S != 3) return cudaErrorInvalidValue;
        SN_DT_SWITCH(dt, T, weight_wino_kernel<T><<<grid_for(K * Cg, 256), 256, 0, st>>>(w, (T *)out, K, Cg));
        return cudaGetLastError();
    }
    if (fmt == W_KRSC_PAD64) {  // rows padded with zeros to a multiple of 64 taps
        const int64_t kpad = (Cg * R * S + 63) / 64 * 64;
        cudaError_t e = cudaMemsetAsync(out, 0, (size_t)K * kpad * dtype_size(dt), st);
        if (e != cudaSuccess) return e;
    }
    SN_DT_SWITCH(dt, T,
                 weight_perm_kernel<T><<<grid_for(K * Cg * R * S, 256), 256, 0, st>>>(w, (T *)out, fmt, K, Cg, R, S));
    return cudaGetLastError();
}

// ===========================================================================
// direct convolution: one output element per thread (the untuned baseline)
// ===========================================================================
template <typename T>
__global__ void conv_direct_nchw(const T *__restrict__ x, const T *__restrict__ w,
                                 const float *__restrict__ bias, T *__restrict__ y, ConvDims d) {
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
        stf<T>(y + i, act_apply(acc + bias[kk], d.act));
    }
}

template <typename T>
__global__ void conv_direct_nhwc(const T *__restrict__ x, const T *__restrict__ w,
                                 const float *__restrict__ bias, T *__restrict__ y, ConvDims d) {
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
        stf<T>(y + i, act_apply(acc + bias[kk], d.act));
    }
}

cudaError_t conv_direct(const LaunchArgs &a) {
    const ConvDims d = conv_dims(a);
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (a.schema.layout == SN_NCHW)
            conv_direct_nchw<T><<<grid_for(total, 256), 256, 0, a.stream>>>(
                (const T *)a.in[0], (const T *)a.wt, a.bias, (T *)a.out, d);
        else
            conv_direct_nhwc<T><<<grid_for(total, 256), 256, 0, a.stream>>>(
                (const T *)a.in[0], (const T *)a.wt, a.bias, (T *)a.out, d);
    });
    return cudaGetLastError();
}

// ===========================================================================
// depthwise convolution
// ===========================================================================
template <typename T>
__global__ void dw_nchw(const T *__restrict__ x, const T *__restrict__ w, const float *__restrict__ bias,
                        T *__restrict__ y, ConvDims d) {
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int q = (int)(i % d.Q), p = (int)((i / d.Q) % d.P);
        const int64_t nc = i / ((int64_t)d.Q * d.P);
        const int c = (int)(nc % d.C);
        const T *xc = x + nc * d.H * (int64_t)d.W;
        const T *wc = w + (int64_t)c * d.R * d.S;
        float acc = 0.f;
        for (int r = 0; r < d.R; ++r) {
            const int h = p * d.sh - d.ph + r * d.dh;
            if (h < 0 || h >= d.H) continue;
            for (int s = 0; s < d.S; ++s) {
                const int ww = q * d.sw - d.pw + s * d.dw;
                if (ww < 0 || ww >= d.W) continue;
                acc += ldf<T>(xc + (int64_t)h * d.W + ww) * ldf<T>(wc + r * d.S + s);
            }
        }
        stf<T>(y + i, act_apply(acc + bias[c], d.act));
    }
}

template <typename T>
__global__ void dw_nhwc(const T *__restrict__ x, const T *__restrict__ w, const float *__restrict__ bias,
                        T *__restrict__ y, ConvDims d) {
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

cudaError_t dwconv(const LaunchArgs &a) {
    const ConvDims d = conv_dims(a);
    const int64_t total = (int64_t)d.N * d.K * d.P * d.Q;
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (a.schema.layout == SN_NCHW)
            dw_nchw<T><<<grid_for(total, 256), 256, 0, a.stream>>>((const T *)a.in[0], (const T *)a.wt,
                                                                    a.bias, (T *)a.out, d);
        else
            dw_nhwc<T><<<grid_for(total, 256), 256, 0, a.stream>>>((const T *)a.in[0], (const T *)a.wt,
                                                                    a.bias, (T *)a.out, d);
    });
    return cudaGetLastError();
}

// ===========================================================================
// max pooling (-inf padding), global average pooling, add, dense
// ===========================================================================
template <typename T, bool NHWC>
__global__ void maxpool_kernel(const T *__restrict__ x, T *__restrict__ y, int N, int C, int H, int W,
                               int P, int Q, int kh, int kw, int sh, int sw, int ph, int pw) {
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
template <typename T>
__global__ void maxpool_nhwc_vec(const uint4 *__restrict__ x, uint4 *__restrict__ y, int N, int C16, int H, int W,
                                 int P, int Q, int kh, int kw, int sh, int sw, int ph, int pw) {
    constexpr int E = 16 / sizeof(T);
    const int64_t total = (int64_t)N * P * Q * C16;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int cv = (int)(i % C16);
        const int64_t pix = i / C16;
        const int q = (int)(pix % Q), p = (int)((pix / Q) % P);
        const int64_t n = pix / ((int64_t)Q * P);
        float m[E];
#pragma unroll
        for (int e = 0; e < E; ++e) m[e] = -INFINITY;
        for (int r = 0; r < kh; ++r) {
            const int h = p * sh - ph + r;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < kw; ++s) {
                const int ww = q * sw - pw + s;
                if (ww < 0 || ww >= W) continue;
                const uint4 v = x[((n * H + h) * W + ww) * C16 + cv];
                const T *pv = reinterpret_cast<const T *>(&v);
#pragma unroll
                for (int e = 0; e < E; ++e) m[e] = fmaxf(m[e], ldf<T>(pv + e));
            }
        }
        uint4 o;
        T *po = reinterpret_cast<T *>(&o);
#pragma unroll
        for (int e = 0; e < E; ++e) po[e] = cvt<T>(m[e]);  // exact: m is one of the stored values
        y[i] = o;
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
            maxpool_nhwc_vec<T><<<grid_for(o.n * o.h * o.w * c16, 256), 256, 0, a.stream>>>(
                (const uint4 *)a.in[0], (uint4 *)a.out, (int)i.n, c16, (int)i.h, (int)i.w, (int)o.h, (int)o.w,
                p.kh, p.kw, p.sh, p.sw, p.ph, p.pw);
        } else if (a.schema.layout == SN_NHWC)
            maxpool_kernel<T, true><<<grid_for(total, 256), 256, 0, a.stream>>>(
                (const T *)a.in[0], (T *)a.out, (int)i.n, (int)i.c, (int)i.h, (int)i.w, (int)o.h, (int)o.w,
                p.kh, p.kw, p.sh, p.sw, p.ph, p.pw);
        else
            maxpool_kernel<T, false><<<grid_for(total, 256), 256, 0, a.stream>>>(
                (const T *)a.in[0], (T *)a.out, (int)i.n, (int)i.c, (int)i.h, (int)i.w, (int)o.h, (int)o.w,
                p.kh, p.kw, p.sh, p.sw, p.ph, p.pw);
    });
    return cudaGetLastError();
}

// NCHW: one warp per (n, c) sums HW contiguous values
template <typename T>
__global__ void gap_nchw(const T *__restrict__ x, T *__restrict__ y, int64_t NC, int64_t HW) {
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / 32;
    const int lane = threadIdx.x % 32;
    for (int64_t nc = warp; nc < NC; nc += (int64_t)gridDim.x * blockDim.x / 32) {
        float s = 0.f;
        for (int64_t i = lane; i < HW; i += 32) s += ldf<T>(x + nc * HW + i);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) stf<T>(y + nc, s / (float)HW);
    }
}

// NHWC: one thread per (n, c); consecutive threads read consecutive channels
template <typename T>
__global__ void gap_nhwc(const T *__restrict__ x, T *__restrict__ y, int64_t N, int64_t C, int64_t HW) {
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
            gap_nchw<T><<<grid_for(i.n * i.c * 32, 256), 256, 0, a.stream>>>((const T *)a.in[0], (T *)a.out,
                                                                               i.n * i.c, i.h * i.w);
        else
            gap_nhwc<T><<<grid_for(i.n * i.c, 256), 256, 0, a.stream>>>((const T *)a.in[0], (T *)a.out, i.n,
                                                                         i.c, i.h * i.w);
    });
    return cudaGetLastError();
}

template <typename T>
__global__ void add_kernel(const T *__restrict__ a, const T *__restrict__ b, T *__restrict__ y, int64_t n,
                           int act) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        stf<T>(y + i, act_apply(ldf<T>(a + i) + ldf<T>(b + i), act));
}

// 8 x 16-bit lanes per thread when everything is 16-byte aligned
template <typename T>
__global__ void add16_kernel(const uint4 *__restrict__ a, const uint4 *__restrict__ b, uint4 *__restrict__ y,
                             int64_t n16, int act) {
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
            add16_kernel<T><<<grid_for(bytes / 16, 256), 256, 0, a.stream>>>(
                (const uint4 *)a.in[0], (const uint4 *)a.in[1], (uint4 *)a.out, bytes / 16, a.layer->act);
        else
            add_kernel<T><<<grid_for(n, 256), 256, 0, a.stream>>>((const T *)a.in[0], (const T *)a.in[1],
                                                                   (T *)a.out, n, a.layer->act);
    });
    return cudaGetLastError();
}

// dense: one warp per (n, o), dot product over the input features
template <typename T>
__global__ void dense_kernel(const T *__restrict__ x, const T *__restrict__ w, const float *__restrict__ bias,
                             T *__restrict__ y, int64_t N, int64_t IN, int64_t OUT, int act) {
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
                 dense_kernel<T><<<grid_for(N * OUT * 32, 256), 256, 0, a.stream>>>(
                     (const T *)a.in[0], (const T *)a.wt, a.bias, (T *)a.out, N, IN, OUT, a.layer->act));
    return cudaGetLastError();
}

}  // namespace k
}  // namespace sn
