// Allocation-free Winograd convolution (declared in include/sn.h as
// sn_conv2d_wino_noalloc).  The paper has no counterpart: this entry point is
// for callers that may not allocate device memory when they run a layer.
//
// Its scratch is one file-scope device array of SN_NOALLOC_SCRATCH_BYTES.
// Host code cannot use the array's name as a device address (on the host it
// names a stand-in object), so the first call on each device looks up the
// real address with cudaGetSymbolAddress while that device is current and
// caches it; later calls reuse it.  Nothing here calls cudaMalloc/cudaFree or
// the graph's allocator hooks.
#include <mutex>
#include <string>

#include "kern_common.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[SN_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_ptr[kMaxDevices] = {};

// device address of the scratch array on the current device (set-up on first use)
sn_status scratch_on_current_device(void **out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return sn::fail(SN_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices) return sn::fail(SN_EUNSUPPORTED, "device index beyond the scratch table");
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return sn::fail(SN_ECUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return SN_OK;
}

size_t align256(size_t v) { return (v + 255) & ~size_t(255); }

}  // namespace

extern "C" sn_status sn_conv2d_wino_noalloc(const void *x_dev, sn_schema schema, const int64_t in_nchw[4],
                                            int32_t c_out, int32_t pad, int32_t act, const float *w_dev,
                                            const float *bias_dev, void *y_dev, void *stream) {
    try {
        using namespace sn;
        if (!x_dev || !in_nchw || !w_dev || !bias_dev || !y_dev)
            return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: NULL argument");
        if (!schema_valid(schema)) return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: invalid schema");
        if (schema.dtype == SN_QI8)
            return fail(SN_EUNSUPPORTED, "sn_conv2d_wino_noalloc: the Winograd routine has no qint8 form");
        if (pad < 0 || pad > 2) return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: pad must be 0, 1 or 2");
        if (act < SN_ACT_NONE || act > SN_ACT_HSIGMOID) return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: bad act");
        for (int i = 0; i < 4; ++i)
            if (in_nchw[i] < 1 || in_nchw[i] > (1 << 30))
                return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: extents must be in [1, 2^30]");
        if (c_out < 1) return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: c_out must be >= 1");
        const int64_t N = in_nchw[0], C = in_nchw[1], H = in_nchw[2], W = in_nchw[3];
        const int64_t P = H + 2 * pad - 2, Q = W + 2 * pad - 2;
        if (P < 1 || Q < 1) return fail(SN_EINVAL, "sn_conv2d_wino_noalloc: empty output");
        // Every byte count is a product of extents of up to 2^30 each, so it
        // is formed with overflow checks: a count that does not fit in 64
        // bits is far beyond the scratch size and is rejected as such.
        const uint64_t limit = SN_NOALLOC_SCRATCH_BYTES;
        auto mul = [](uint64_t a, uint64_t b, uint64_t *out) { return !__builtin_mul_overflow(a, b, out); };
        uint64_t tiles = 0, u_raw = 0, v_raw = 0, m_raw = 0, need = 0;
        const bool in64 =
            mul((uint64_t)N, (uint64_t)((P + 1) / 2), &tiles) && mul(tiles, (uint64_t)((Q + 1) / 2), &tiles) &&
            mul((uint64_t)16 * dtype_size(schema.dtype), (uint64_t)c_out, &u_raw) && mul(u_raw, (uint64_t)C, &u_raw) &&
            mul((uint64_t)16 * sizeof(float), tiles, &v_raw) && mul(v_raw, (uint64_t)C, &v_raw) &&
            mul((uint64_t)16 * sizeof(float), tiles, &m_raw) && mul(m_raw, (uint64_t)c_out, &m_raw) &&
            !__builtin_add_overflow(u_raw, v_raw, &need) && !__builtin_add_overflow(need, m_raw, &need);
        // each part is rounded up to 256 bytes: at most 3 x 255 more than `need`
        if (!in64 || need > limit || align256(u_raw) + align256(v_raw) + align256(m_raw) > limit)
            return fail(SN_EUNSUPPORTED, "sn_conv2d_wino_noalloc: needs " +
                                             (in64 ? std::to_string(need) : std::string("more than 2^64")) +
                                             " bytes of scratch, the fixed limit is " + std::to_string(limit));
        const size_t u_bytes = align256(u_raw), v_bytes = align256(v_raw);
        void *scratch = nullptr;
        sn_status rc = scratch_on_current_device(&scratch);
        if (rc != SN_OK) return rc;
        unsigned char *base = static_cast<unsigned char *>(scratch);
        void *U = base;
        float *V = reinterpret_cast<float *>(base + u_bytes);
        float *Mx = reinterpret_cast<float *>(base + u_bytes + v_bytes);
        cudaStream_t st = static_cast<cudaStream_t>(stream);
        // U = G g G^T from the caller's fp32 weights (every element written)
        cudaError_t e = k::weight_format(w_dev, U, k::W_WINO, schema.dtype, c_out, C, 3, 3, st);
        if (e == cudaSuccess) {
            const k::ConvDims d{(int32_t)N, (int32_t)C, (int32_t)H, (int32_t)W, c_out, (int32_t)P, (int32_t)Q,
                                3, 3, 1, 1, pad, pad, 1, 1, 1, act};
            e = k::conv_wino_buffers(d, schema, x_dev, U, bias_dev, y_dev, V, Mx, st);
        }
        if (e != cudaSuccess)
            return fail(SN_ECUDA, std::string("sn_conv2d_wino_noalloc: ") + cudaGetErrorString(e));
        return SN_OK;
    } catch (...) {
        return sn::fail(SN_EINVAL, "sn_conv2d_wino_noalloc: internal error");
    }
}
