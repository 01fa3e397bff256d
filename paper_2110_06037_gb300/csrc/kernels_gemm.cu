// Convolution as GEMM on CUDA cores:
//   * implicit GEMM (M = N*P*Q output pixels, N = K output channels,
//     K = C*R*S taps), the im2col gather done on the fly while staging tiles
//     in shared memory, register-tiled FFMA, fused bias + activation;
//   * Winograd F(2x2,3x3) as a childnet of three sub-layers (section III-D):
//     wgenc (V = B^T d B per 4x4 input tile), wgconv (16 batched GEMMs
//     M_xi = V_xi U_xi^T), wgdec (Y = A^T M A per 2x2 output tile + bias +
//     activation).  The filter transform U = G g G^T is done once when the
//     weights are prepared.
#include "kern_common.cuh"

namespace sn {
namespace k {

// ---------------------------------------------------------------------------
// implicit GEMM, BM x 64 x 16 tiles, 256 threads, (BM/16) x 4 outputs each
// ---------------------------------------------------------------------------
template <typename T, bool NHWC, int BM>
__global__ void __launch_bounds__(256) igemm_simt_kernel(const T *__restrict__ x, const T *__restrict__ w,
                                                         const float *__restrict__ bias, T *__restrict__ y,
                                                         ConvDims d) {
    griddep_launch();
    griddep_wait();
    constexpr int BN = 64, BK = 16, TM = BM / 16, TN = 4;
    constexpr int A_PER = BK * BM / 256, B_PER = BK * BN / 256;
    __shared__ float As[BK][BM + 4];
    __shared__ float Bs[BK][BN + 4];
    __shared__ int64_t m_base[BM];
    __shared__ int m_h0[BM], m_w0[BM];

    const int tid = threadIdx.x;
    const int64_t M = (int64_t)d.N * d.P * d.Q;
    const int PQ = d.P * d.Q, RS = d.R * d.S;
    const int Kg = d.C * RS;
    const int64_t m0 = (int64_t)blockIdx.x * BM;
    const int n0 = blockIdx.y * BN;

    for (int m = tid; m < BM; m += 256) {
        const int64_t mg = m0 + m;
        if (mg < M) {
            const int64_t n = mg / PQ;
            const int pq = (int)(mg % PQ), p = pq / d.Q, q = pq % d.Q;
            m_base[m] = n * (int64_t)d.C * d.H * d.W;
            m_h0[m] = p * d.sh - d.ph;
            m_w0[m] = q * d.sw - d.pw;
        } else {
            m_base[m] = 0;
            m_h0[m] = -(1 << 28);  // every tap out of bounds
            m_w0[m] = 0;
        }
    }
    __syncthreads();

    const int tm = NHWC ? tid / 16 : tid % 16;
    const int tn = NHWC ? tid % 16 : tid / 16;
    float acc[TM][TN];
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

    float ra[A_PER], rb[B_PER];
    auto load = [&](int k0) {
#pragma unroll
        for (int it = 0; it < A_PER; ++it) {
            const int e = tid + it * 256;
            const int m = NHWC ? e / BK : e % BM;
            const int kk = NHWC ? e % BK : e / BM;
            const int kg = k0 + kk;
            float v = 0.f;
            if (kg < Kg) {
                int c, r, s;
                if (NHWC) {
                    c = kg % d.C;
                    const int rs = kg / d.C;
                    r = rs / d.S;
                    s = rs % d.S;
                } else {
                    c = kg / RS;
                    const int rs = kg % RS;
                    r = rs / d.S;
                    s = rs % d.S;
                }
                const int h = m_h0[m] + r * d.dh, ww = m_w0[m] + s * d.dw;
                if (h >= 0 && h < d.H && ww >= 0 && ww < d.W) {
                    const int64_t idx = NHWC ? m_base[m] + ((int64_t)h * d.W + ww) * d.C + c
                                             : m_base[m] + ((int64_t)c * d.H + h) * d.W + ww;
                    v = ldf<T>(x + idx);
                }
            }
            ra[it] = v;
        }
#pragma unroll
        for (int it = 0; it < B_PER; ++it) {
            const int e = tid + it * 256;
            const int kk = e % BK, j = e / BK;
            const int kg = k0 + kk, kn = n0 + j;
            rb[it] = (kg < Kg && kn < d.K) ? ldf<T>(w + (int64_t)kn * Kg + kg) : 0.f;
        }
    };
    auto store = [&]() {
#pragma unroll
        for (int it = 0; it < A_PER; ++it) {
            const int e = tid + it * 256;
            const int m = NHWC ? e / BK : e % BM;
            const int kk = NHWC ? e % BK : e / BM;
            As[kk][m] = ra[it];
        }
#pragma unroll
        for (int it = 0; it < B_PER; ++it) {
            const int e = tid + it * 256;
            Bs[e % BK][e / BK] = rb[it];
        }
    };

    load(0);
    for (int k0 = 0; k0 < Kg; k0 += BK) {
        store();
        __syncthreads();
        if (k0 + BK < Kg) load(k0 + BK);  // overlaps the global loads with the FMAs below
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float a[TM], b[TN];
#pragma unroll
            for (int i = 0; i < TM; ++i) a[i] = As[kk][tm + 16 * i];
#pragma unroll
            for (int j = 0; j < TN; ++j) b[j] = Bs[kk][tn + 16 * j];
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }

#pragma unroll
    for (int i = 0; i < TM; ++i) {
        const int64_t mg = m0 + tm + 16 * i;
        if (mg >= M) continue;
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int kn = n0 + tn + 16 * j;
            if (kn >= d.K) continue;
            const float v = act_apply(acc[i][j] + bias[kn], d.act);
            int64_t o;
            if (NHWC) {
                o = mg * d.K + kn;
            } else {
                const int64_t n = mg / PQ;
                o = (n * d.K + kn) * PQ + (mg % PQ);
            }
            stf<T>(y + o, v);
        }
    }
}

cudaError_t conv_igemm(const LaunchArgs &a) {
    const ConvDims d = conv_dims(a);
    if (d.groups != 1) return cudaErrorInvalidValue;
    const int64_t M = (int64_t)d.N * d.P * d.Q;
    const int BM = a.variant == 0 ? 64 : 128;
    dim3 grid((unsigned)((M + BM - 1) / BM), (unsigned)((d.K + 63) / 64));
    if (grid.y > 65535) return cudaErrorInvalidValue;
    SN_DT_SWITCH(a.schema.dtype, T, {
        const T *x = (const T *)a.in[0];
        const T *w = (const T *)a.wt;
        T *y = (T *)a.out;
        if (a.schema.layout == SN_NHWC) {
            if (BM == 64) launch_pdl(igemm_simt_kernel<T, true, 64>, grid, 256, 0, a.stream, x, w, a.bias, y, d);
            else launch_pdl(igemm_simt_kernel<T, true, 128>, grid, 256, 0, a.stream, x, w, a.bias, y, d);
        } else {
            if (BM == 64) launch_pdl(igemm_simt_kernel<T, false, 64>, grid, 256, 0, a.stream, x, w, a.bias, y, d);
            else launch_pdl(igemm_simt_kernel<T, false, 128>, grid, 256, 0, a.stream, x, w, a.bias, y, d);
        }
    });
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Winograd F(2x2, 3x3)
// ---------------------------------------------------------------------------
struct WinoDims {
    ConvDims d;
    int tP, tQ;  // output tiles per image along H and W
    int64_t T;   // total tiles N * tP * tQ
};

static WinoDims wino_dims(const ConvDims &d) {
    WinoDims w;
    w.d = d;
    w.tP = (d.P + 1) / 2;
    w.tQ = (d.Q + 1) / 2;
    w.T = (int64_t)d.N * w.tP * w.tQ;
    return w;
}

size_t conv_wino_ws(const Layer &l, const Shape &in, sn_schema s) {
    (void)s;
    const int64_t tiles = in.n * ((l.out.h + 1) / 2) * ((l.out.w + 1) / 2);
    return (size_t)16 * tiles * (in.c + l.out.c) * sizeof(float);
}

// wgenc: V[xi][t][c] = (B^T d B)[xi] for the 4x4 input tile of output tile t
template <typename T, bool NHWC>
__global__ void wino_input_kernel(const T *__restrict__ x, float *__restrict__ V, WinoDims wd) {
    griddep_launch();
    griddep_wait();
    const ConvDims &d = wd.d;
    const int64_t total = wd.T * d.C;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % d.C);
        const int64_t t = i / d.C;
        const int tq = (int)(t % wd.tQ), tp = (int)((t / wd.tQ) % wd.tP);
        const int64_t n = t / ((int64_t)wd.tQ * wd.tP);
        const int h0 = 2 * tp - d.ph, w0 = 2 * tq - d.pw;
        float v[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const int h = h0 + a, ww = w0 + b;
                float val = 0.f;
                if (h >= 0 && h < d.H && ww >= 0 && ww < d.W) {
                    const int64_t idx = NHWC ? ((n * d.H + h) * d.W + ww) * d.C + c
                                             : ((n * d.C + c) * d.H + h) * (int64_t)d.W + ww;
                    val = ldf<T>(x + idx);
                }
                v[a][b] = val;
            }
        float t4[4][4];  // B^T d
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            t4[0][b] = v[0][b] - v[2][b];
            t4[1][b] = v[1][b] + v[2][b];
            t4[2][b] = v[2][b] - v[1][b];
            t4[3][b] = v[1][b] - v[3][b];
        }
#pragma unroll
        for (int a = 0; a < 4; ++a) {  // (B^T d) B
            const float o[4] = {t4[a][0] - t4[a][2], t4[a][1] + t4[a][2], t4[a][2] - t4[a][1],
                                t4[a][1] - t4[a][3]};
#pragma unroll
            for (int b = 0; b < 4; ++b) V[((int64_t)(a * 4 + b) * wd.T + t) * d.C + c] = o[b];
        }
    }
}

// wgconv: Mx[b][m][n] = sum_k A[b][m][k] * B[b][n][k]; A fp32, B of type TB
template <typename TB>
__global__ void __launch_bounds__(256) gemm_nt_simt(const float *__restrict__ A, const TB *__restrict__ B,
                                                    float *__restrict__ Cm, int64_t M, int N, int Kd) {
    griddep_launch();
    griddep_wait();
    constexpr int BM = 64, BN = 64, BK = 16, TM = 4, TN = 4;
    __shared__ float As[BK][BM + 4];
    __shared__ float Bs[BK][BN + 4];
    const int b = blockIdx.z;
    const float *Ab = A + (int64_t)b * M * Kd;
    const TB *Bb = B + (int64_t)b * N * Kd;
    float *Cb = Cm + (int64_t)b * M * N;
    const int tid = threadIdx.x, tm = tid / 16, tn = tid % 16;
    const int64_t m0 = (int64_t)blockIdx.x * BM;
    const int n0 = blockIdx.y * BN;
    float acc[TM][TN] = {};
    for (int k0 = 0; k0 < Kd; k0 += BK) {
#pragma unroll
        for (int it = 0; it < 4; ++it) {
            const int e = tid + it * 256, kk = e % BK, r = e / BK;
            const int64_t mg = m0 + r;
            const int ng = n0 + r, kg = k0 + kk;
            As[kk][r] = (mg < M && kg < Kd) ? Ab[mg * Kd + kg] : 0.f;
            Bs[kk][r] = (ng < N && kg < Kd) ? ldf<TB>(Bb + (int64_t)ng * Kd + kg) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float a[TM], bb[TN];
#pragma unroll
            for (int i = 0; i < TM; ++i) a[i] = As[kk][tm + 16 * i];
#pragma unroll
            for (int j = 0; j < TN; ++j) bb[j] = Bs[kk][tn + 16 * j];
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], bb[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < TM; ++i) {
        const int64_t mg = m0 + tm + 16 * i;
        if (mg >= M) continue;
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int ng = n0 + tn + 16 * j;
            if (ng < N) Cb[mg * N + ng] = acc[i][j];
        }
    }
}

// wgdec: Y = A^T M A for each output tile, + bias, activation, store
template <typename T, bool NHWC>
__global__ void wino_output_kernel(const float *__restrict__ Mx, const float *__restrict__ bias,
                                   T *__restrict__ y, WinoDims wd) {
    griddep_launch();
    griddep_wait();
    const ConvDims &d = wd.d;
    const int64_t total = wd.T * d.K;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int kk = (int)(i % d.K);
        const int64_t t = i / d.K;
        const int tq = (int)(t % wd.tQ), tp = (int)((t / wd.tQ) % wd.tP);
        const int64_t n = t / ((int64_t)wd.tQ * wd.tP);
        float m[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) m[a][b] = Mx[((int64_t)(a * 4 + b) * wd.T + t) * d.K + kk];
        float u[2][4];  // A^T M
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            u[0][b] = m[0][b] + m[1][b] + m[2][b];
            u[1][b] = m[1][b] - m[2][b] - m[3][b];
        }
        const float bv = bias[kk];
#pragma unroll
        for (int a = 0; a < 2; ++a) {
            const float yy[2] = {u[a][0] + u[a][1] + u[a][2], u[a][1] - u[a][2] - u[a][3]};
            const int p = 2 * tp + a;
            if (p >= d.P) continue;
#pragma unroll
            for (int b = 0; b < 2; ++b) {
                const int q = 2 * tq + b;
                if (q >= d.Q) continue;
                const int64_t o = NHWC ? ((n * d.P + p) * d.Q + q) * d.K + kk
                                       : ((n * d.K + kk) * d.P + p) * (int64_t)d.Q + q;
                stf<T>(y + o, act_apply(yy[b] + bv, d.act));
            }
        }
    }
}

cudaError_t conv_wino(const LaunchArgs &a) { return conv_wino_stage(a, -1); }

// stage 0: input transform (wgenc); 1: element-wise GEMMs (wgconv); 2: output
// transform (wgdec); -1: all three
cudaError_t conv_wino_stage(const LaunchArgs &a, int stage) {
    const ConvDims d = conv_dims(a);
    const WinoDims wd = wino_dims(d);
    const size_t need = (size_t)16 * wd.T * (d.C + d.K) * sizeof(float);
    if (!a.ws || a.ws_bytes < need) return cudaErrorInvalidValue;
    float *V = static_cast<float *>(a.ws);
    float *Mx = V + (size_t)16 * wd.T * d.C;
    dim3 ggrid((unsigned)((wd.T + 63) / 64), (unsigned)((d.K + 63) / 64), 16);
    if (ggrid.y > 65535) return cudaErrorInvalidValue;
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (stage < 0 || stage == 0) {
            if (a.schema.layout == SN_NHWC)
                launch_pdl(wino_input_kernel<T, true>, grid_for(wd.T * d.C, 256), 256, 0, a.stream, (const T *)a.in[0], V, wd);
            else
                launch_pdl(wino_input_kernel<T, false>, grid_for(wd.T * d.C, 256), 256, 0, a.stream, (const T *)a.in[0], V, wd);
        }
        if (stage < 0 || stage == 1) {
            launch_pdl(gemm_nt_simt<T>, ggrid, 256, 0, a.stream, V, (const T *)a.wt, Mx, wd.T, d.K, d.C);
        }
        if (stage < 0 || stage == 2) {
            if (a.schema.layout == SN_NHWC)
                launch_pdl(wino_output_kernel<T, true>, grid_for(wd.T * d.K, 256), 256, 0, a.stream, Mx, a.bias, (T *)a.out, wd);
            else
                launch_pdl(wino_output_kernel<T, false>, grid_for(wd.T * d.K, 256), 256, 0, a.stream, Mx, a.bias, (T *)a.out, wd);
        }
    });
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Winograd F(4x4, 3x3): 6x6 input tiles, 36 element-wise GEMMs, 4x4 outputs
// (Lavin & Gray's interpolation points 0, +-1, +-2 and infinity).  The
// transformed filters are kept in fp32 whatever the schema (the larger
// transform coefficients would amplify a 16-bit rounding of U).
// ---------------------------------------------------------------------------
static WinoDims wino4_dims(const ConvDims &d) {
    WinoDims w;
    w.d = d;
    w.tP = (d.P + 3) / 4;
    w.tQ = (d.Q + 3) / 4;
    w.T = (int64_t)d.N * w.tP * w.tQ;
    return w;
}

size_t conv_wino4_ws(const Layer &l, const Shape &in, sn_schema s) {
    (void)s;
    const int64_t tiles = in.n * ((l.out.h + 3) / 4) * ((l.out.w + 3) / 4);
    return (size_t)36 * tiles * (in.c + l.out.c) * sizeof(float);
}

// r = B^T d for one column d of the 6x6 tile
__device__ __forceinline__ void wino4_bt(const float (&d)[6], float (&r)[6]) {
    r[0] = 4.f * d[0] - 5.f * d[2] + d[4];
    r[1] = -4.f * d[1] - 4.f * d[2] + d[3] + d[4];
    r[2] = 4.f * d[1] - 4.f * d[2] - d[3] + d[4];
    r[3] = -2.f * d[1] - d[2] + 2.f * d[3] + d[4];
    r[4] = 2.f * d[1] - d[2] - 2.f * d[3] + d[4];
    r[5] = 4.f * d[1] - 5.f * d[3] + d[5];
}
// o = A^T m for one column m
__device__ __forceinline__ void wino4_at(const float (&m)[6], float (&o)[4]) {
    o[0] = m[0] + m[1] + m[2] + m[3] + m[4];
    o[1] = m[1] - m[2] + 2.f * (m[3] - m[4]);
    o[2] = m[1] + m[2] + 4.f * (m[3] + m[4]);
    o[3] = m[1] - m[2] + 8.f * (m[3] - m[4]) + m[5];
}

// wgenc: V[xi][t][c] = (B^T d B)[xi] for the 6x6 input tile of output tile t
template <typename T, bool NHWC>
__global__ void wino4_input_kernel(const T *__restrict__ x, float *__restrict__ V, WinoDims wd) {
    griddep_launch();
    griddep_wait();
    const ConvDims &d = wd.d;
    const int64_t total = wd.T * d.C;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % d.C);
        const int64_t t = i / d.C;
        const int tq = (int)(t % wd.tQ), tp = (int)((t / wd.tQ) % wd.tP);
        const int64_t n = t / ((int64_t)wd.tQ * wd.tP);
        const int h0 = 4 * tp - d.ph, w0 = 4 * tq - d.pw;
        float v[6][6];
#pragma unroll
        for (int a = 0; a < 6; ++a)
#pragma unroll
            for (int b = 0; b < 6; ++b) {
                const int h = h0 + a, ww = w0 + b;
                float val = 0.f;
                if (h >= 0 && h < d.H && ww >= 0 && ww < d.W) {
                    const int64_t idx = NHWC ? ((n * d.H + h) * d.W + ww) * d.C + c
                                             : ((n * d.C + c) * d.H + h) * (int64_t)d.W + ww;
                    val = ldf<T>(x + idx);
                }
                v[a][b] = val;
            }
        float t6[6][6];  // B^T d, column by column
#pragma unroll
        for (int b = 0; b < 6; ++b) {
            const float col[6] = {v[0][b], v[1][b], v[2][b], v[3][b], v[4][b], v[5][b]};
            float r[6];
            wino4_bt(col, r);
#pragma unroll
            for (int a = 0; a < 6; ++a) t6[a][b] = r[a];
        }
#pragma unroll
        for (int a = 0; a < 6; ++a) {  // (B^T d) B: B^T applied to each row
            float r[6];
            wino4_bt(t6[a], r);
#pragma unroll
            for (int b = 0; b < 6; ++b) V[((int64_t)(a * 6 + b) * wd.T + t) * d.C + c] = r[b];
        }
    }
}

// wgdec: Y = A^T M A for each output tile, + bias, activation, store
template <typename T, bool NHWC>
__global__ void wino4_output_kernel(const float *__restrict__ Mx, const float *__restrict__ bias,
                                    T *__restrict__ y, WinoDims wd) {
    griddep_launch();
    griddep_wait();
    const ConvDims &d = wd.d;
    const int64_t total = wd.T * d.K;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int kk = (int)(i % d.K);
        const int64_t t = i / d.K;
        const int tq = (int)(t % wd.tQ), tp = (int)((t / wd.tQ) % wd.tP);
        const int64_t n = t / ((int64_t)wd.tQ * wd.tP);
        float u[4][6];  // A^T M, column by column
#pragma unroll
        for (int b = 0; b < 6; ++b) {
            float col[6];
#pragma unroll
            for (int a = 0; a < 6; ++a) col[a] = Mx[((int64_t)(a * 6 + b) * wd.T + t) * d.K + kk];
            float o[4];
            wino4_at(col, o);
#pragma unroll
            for (int a = 0; a < 4; ++a) u[a][b] = o[a];
        }
        const float bv = bias[kk];
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            const int p = 4 * tp + a;
            if (p >= d.P) continue;
            float yy[4];
            wino4_at(u[a], yy);
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const int q = 4 * tq + b;
                if (q >= d.Q) continue;
                const int64_t o = NHWC ? ((n * d.P + p) * d.Q + q) * d.K + kk
                                       : ((n * d.K + kk) * d.P + p) * (int64_t)d.Q + q;
                stf<T>(y + o, act_apply(yy[b] + bv, d.act));
            }
        }
    }
}

cudaError_t conv_wino4(const LaunchArgs &a) { return conv_wino4_stage(a, -1); }

// stage 0: input transform (wgenc); 1: element-wise GEMMs (wgconv); 2: output
// transform (wgdec); -1: all three
cudaError_t conv_wino4_stage(const LaunchArgs &a, int stage) {
    const ConvDims d = conv_dims(a);
    const WinoDims wd = wino4_dims(d);
    const size_t need = (size_t)36 * wd.T * (d.C + d.K) * sizeof(float);
    if (!a.ws || a.ws_bytes < need) return cudaErrorInvalidValue;
    float *V = static_cast<float *>(a.ws);
    float *Mx = V + (size_t)36 * wd.T * d.C;
    dim3 ggrid((unsigned)((wd.T + 63) / 64), (unsigned)((d.K + 63) / 64), 36);
    if (ggrid.y > 65535) return cudaErrorInvalidValue;
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (stage < 0 || stage == 0) {
            if (a.schema.layout == SN_NHWC)
                launch_pdl(wino4_input_kernel<T, true>, grid_for(wd.T * d.C, 256), 256, 0, a.stream, (const T *)a.in[0],
                           V, wd);
            else
                launch_pdl(wino4_input_kernel<T, false>, grid_for(wd.T * d.C, 256), 256, 0, a.stream,
                           (const T *)a.in[0], V, wd);
        }
        if (stage < 0 || stage == 1) {
            launch_pdl(gemm_nt_simt<float>, ggrid, 256, 0, a.stream, V, (const float *)a.wt, Mx, wd.T, d.K, d.C);
        }
        if (stage < 0 || stage == 2) {
            if (a.schema.layout == SN_NHWC)
                launch_pdl(wino4_output_kernel<T, true>, grid_for(wd.T * d.K, 256), 256, 0, a.stream, Mx, a.bias,
                           (T *)a.out, wd);
            else
                launch_pdl(wino4_output_kernel<T, false>, grid_for(wd.T * d.K, 256), 256, 0, a.stream, Mx, a.bias,
                           (T *)a.out, wd);
        }
    });
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Winograd F(6x6, 3x3): 8x8 input tiles, 64 element-wise GEMMs, 6x6 outputs
// (Toom-Cook interpolation points 0, +-1, +-2, +-1/2 and infinity; the
// paper's tile_size 8).  Transformed filters and the GEMM stay fp32.
// ---------------------------------------------------------------------------
static WinoDims wino6_dims(const ConvDims &d) {
    WinoDims w;
    w.d = d;
    w.tP = (d.P + 5) / 6;
    w.tQ = (d.Q + 5) / 6;
    w.T = (int64_t)d.N * w.tP * w.tQ;
    return w;
}

size_t conv_wino6_ws(const Layer &l, const Shape &in, sn_schema s) {
    (void)s;
    const int64_t tiles = in.n * ((l.out.h + 5) / 6) * ((l.out.w + 5) / 6);
    return (size_t)64 * tiles * (in.c + l.out.c) * sizeof(float);
}

// r = B^T d for one column d of the 8x8 tile
__device__ __forceinline__ void wino6_bt(const float (&d)[8], float (&r)[8]) {
    r[0] = d[0] - 5.25f * d[2] + 5.25f * d[4] - d[6];
    r[1] = d[1] + d[2] - 4.25f * d[3] - 4.25f * d[4] + d[5] + d[6];
    r[2] = -d[1] + d[2] + 4.25f * d[3] - 4.25f * d[4] - d[5] + d[6];
    r[3] = 0.5f * d[1] + 0.25f * d[2] - 2.5f * d[3] - 1.25f * d[4] + 2.f * d[5] + d[6];
    r[4] = -0.5f * d[1] + 0.25f * d[2] + 2.5f * d[3] - 1.25f * d[4] - 2.f * d[5] + d[6];
    r[5] = 2.f * d[1] + 4.f * d[2] - 2.5f * d[3] - 5.f * d[4] + 0.5f * d[5] + d[6];
    r[6] = -2.f * d[1] + 4.f * d[2] + 2.5f * d[3] - 5.f * d[4] - 0.5f * d[5] + d[6];
    r[7] = -d[1] + 5.25f * d[3] - 5.25f * d[5] + d[7];
}
// o = A^T m for one column m
__device__ __forceinline__ void wino6_at(const float (&m)[8], float (&o)[6]) {
    const float p12 = m[1] + m[2], m12 = m[1] - m[2];
    const float p34 = m[3] + m[4], m34 = m[3] - m[4];
    const float p56 = m[5] + m[6], m56 = m[5] - m[6];
    o[0] = m[0] + p12 + p34 + p56;
    o[1] = m12 + 2.f * m34 + 0.5f * m56;
    o[2] = p12 + 4.f * p34 + 0.25f * p56;
    o[3] = m12 + 8.f * m34 + 0.125f * m56;
    o[4] = p12 + 16.f * p34 + 0.0625f * p56;
    o[5] = m12 + 32.f * m34 + 0.03125f * m56 + m[7];
}

// wgenc: V[xi][t][c] = (B^T d B)[xi] for the 8x8 input tile of output tile t
template <typename T, bool NHWC>
__global__ void wino6_input_kernel(const T *__restrict__ x, float *__restrict__ V, WinoDims wd) {
    griddep_launch();
    griddep_wait();
    const ConvDims &d = wd.d;
    const int64_t total = wd.T * d.C;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % d.C);
        const int64_t t = i / d.C;
        const int tq = (int)(t % wd.tQ), tp = (int)((t / wd.tQ) % wd.tP);
        const int64_t n = t / ((int64_t)wd.tQ * wd.tP);
        const int h0 = 6 * tp - d.ph, w0 = 6 * tq - d.pw;
        float t8[8][8];  // B^T d, column by column
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            float col[8];
#pragma unroll
            for (int a = 0; a < 8; ++a) {
                const int h = h0 + a, ww = w0 + b;
                float val = 0.f;
                if (h >= 0 && h < d.H && ww >= 0 && ww < d.W) {
                    const int64_t idx = NHWC ? ((n * d.H + h) * d.W + ww) * d.C + c
                                             : ((n * d.C + c) * d.H + h) * (int64_t)d.W + ww;
                    val = ldf<T>(x + idx);
                }
                col[a] = val;
            }
            float r[8];
            wino6_bt(col, r);
#pragma unroll
            for (int a = 0; a < 8; ++a) t8[a][b] = r[a];
        }
#pragma unroll
        for (int a = 0; a < 8; ++a) {  // (B^T d) B: B^T applied to each row
            float r[8];
            wino6_bt(t8[a], r);
#pragma unroll
            for (int b = 0; b < 8; ++b) V[((int64_t)(a * 8 + b) * wd.T + t) * d.C + c] = r[b];
        }
    }
}

// wgdec: Y = A^T M A for each output tile, + bias, activation, store
template <typename T, bool NHWC>
__global__ void wino6_output_kernel(const float *__restrict__ Mx, const float *__restrict__ bias,
                                    T *__restrict__ y, WinoDims wd) {
    griddep_launch();
    griddep_wait();
    const ConvDims &d = wd.d;
    const int64_t total = wd.T * d.K;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int kk = (int)(i % d.K);
        const int64_t t = i / d.K;
        const int tq = (int)(t % wd.tQ), tp = (int)((t / wd.tQ) % wd.tP);
        const int64_t n = t / ((int64_t)wd.tQ * wd.tP);
        float u[6][8];  // A^T M, column by column
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            float col[8];
#pragma unroll
            for (int a = 0; a < 8; ++a) col[a] = Mx[((int64_t)(a * 8 + b) * wd.T + t) * d.K + kk];
            float o[6];
            wino6_at(col, o);
#pragma unroll
            for (int a = 0; a < 6; ++a) u[a][b] = o[a];
        }
        const float bv = bias[kk];
#pragma unroll
        for (int a = 0; a < 6; ++a) {
            const int p = 6 * tp + a;
            if (p >= d.P) continue;
            float yy[6];
            wino6_at(u[a], yy);
#pragma unroll
            for (int b = 0; b < 6; ++b) {
                const int q = 6 * tq + b;
                if (q >= d.Q) continue;
                const int64_t o = NHWC ? ((n * d.P + p) * d.Q + q) * d.K + kk
                                       : ((n * d.K + kk) * d.P + p) * (int64_t)d.Q + q;
                stf<T>(y + o, act_apply(yy[b] + bv, d.act));
            }
        }
    }
}

cudaError_t conv_wino6(const LaunchArgs &a) { return conv_wino6_stage(a, -1); }

// stage 0: input transform (wgenc); 1: element-wise GEMMs (wgconv); 2: output
// transform (wgdec); -1: all three
cudaError_t conv_wino6_stage(const LaunchArgs &a, int stage) {
    const ConvDims d = conv_dims(a);
    const WinoDims wd = wino6_dims(d);
    const size_t need = (size_t)64 * wd.T * (d.C + d.K) * sizeof(float);
    if (!a.ws || a.ws_bytes < need) return cudaErrorInvalidValue;
    float *V = static_cast<float *>(a.ws);
    float *Mx = V + (size_t)64 * wd.T * d.C;
    dim3 ggrid((unsigned)((wd.T + 63) / 64), (unsigned)((d.K + 63) / 64), 64);
    if (ggrid.y > 65535) return cudaErrorInvalidValue;
    SN_DT_SWITCH(a.schema.dtype, T, {
        if (stage < 0 || stage == 0) {
            if (a.schema.layout == SN_NHWC)
                launch_pdl(wino6_input_kernel<T, true>, grid_for(wd.T * d.C, 256), 256, 0, a.stream, (const T *)a.in[0],
                           V, wd);
            else
                launch_pdl(wino6_input_kernel<T, false>, grid_for(wd.T * d.C, 256), 256, 0, a.stream,
                           (const T *)a.in[0], V, wd);
        }
        if (stage < 0 || stage == 1) {
            launch_pdl(gemm_nt_simt<float>, ggrid, 256, 0, a.stream, V, (const float *)a.wt, Mx, wd.T, d.K, d.C);
        }
        if (stage < 0 || stage == 2) {
            if (a.schema.layout == SN_NHWC)
                launch_pdl(wino6_output_kernel<T, true>, grid_for(wd.T * d.K, 256), 256, 0, a.stream, Mx, a.bias,
                           (T *)a.out, wd);
            else
                launch_pdl(wino6_output_kernel<T, false>, grid_for(wd.T * d.K, 256), 256, 0, a.stream, Mx, a.bias,
                           (T *)a.out, wd);
        }
    });
    return cudaGetLastError();
}

// The three Winograd stages on caller-provided buffers (used by the
// allocation-free entry point): U [16][K][C] in the schema dtype, V and Mx fp32.
cudaError_t conv_wino_buffers(const ConvDims &d, sn_schema s, const void *x, const void *u, const float *bias,
                              void *y, float *V, float *Mx, cudaStream_t st) {
    const WinoDims wd = wino_dims(d);
    dim3 ggrid((unsigned)((wd.T + 63) / 64), (unsigned)((d.K + 63) / 64), 16);
    if (ggrid.y > 65535) return cudaErrorInvalidValue;
    SN_DT_SWITCH(s.dtype, T, {
        if (s.layout == SN_NHWC)
            launch_pdl(wino_input_kernel<T, true>, grid_for(wd.T * d.C, 256), 256, 0, st, (const T *)x, V, wd);
        else
            launch_pdl(wino_input_kernel<T, false>, grid_for(wd.T * d.C, 256), 256, 0, st, (const T *)x, V, wd);
        launch_pdl(gemm_nt_simt<T>, ggrid, 256, 0, st, V, (const T *)u, Mx, wd.T, d.K, d.C);
        if (s.layout == SN_NHWC)
            launch_pdl(wino_output_kernel<T, true>, grid_for(wd.T * d.K, 256), 256, 0, st, Mx, bias, (T *)y, wd);
        else
            launch_pdl(wino_output_kernel<T, false>, grid_for(wd.T * d.K, 256), 256, 0, st, Mx, bias, (T *)y, wd);
    });
    return cudaGetLastError();
}

}  // namespace k
}  // namespace sn
