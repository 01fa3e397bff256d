// Halo-tile instantiations of the tensor-core convolution kernel (tc_conv.cuh):
// 3x3 stride-1 layers, one A box per row of taps; a translation unit of their
// own so that they compile beside the others.
#include "tc_conv.cuh"

namespace sn {
namespace k {
namespace tc {

template <typename T>
static cudaError_t launch_halo_dt(int bn, int g, const CUtensorMap *mA, const CUtensorMap &mB, const CUtensorMap &mY,
                                  const CUtensorMap &mR, const Params &p, cudaStream_t st) {
    if (g == 1 && bn == 64) return launch<T, 64, true, 1, 1, false, 1, 1, false, true>(mA, mB, mY, mR, p, st);
    if (g == 1 && bn == 128) return launch<T, 128, true, 1, 1, false, 1, 1, false, true>(mA, mB, mY, mR, p, st);
    if (g == 2 && bn == 64) return launch<T, 64, true, 2, 1, false, 1, 1, false, true>(mA, mB, mY, mR, p, st);
    if (g == 2 && bn == 128) return launch<T, 128, true, 2, 1, false, 1, 1, false, true>(mA, mB, mY, mR, p, st);
    if (g == 2 && bn == 256) return launch<T, 256, true, 2, 1, false, 1, 1, false, true>(mA, mB, mY, mR, p, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_halo(int dtype, int bn, int g, const CUtensorMap *mA, const CUtensorMap &mB,
                        const CUtensorMap &mY, const CUtensorMap &mR, const Params &p, cudaStream_t st) {
    if (dtype == SN_BF16) return launch_halo_dt<__nv_bfloat16>(bn, g, mA, mB, mY, mR, p, st);
    if (dtype == SN_F16) return launch_halo_dt<__half>(bn, g, mA, mB, mY, mR, p, st);
    return cudaErrorInvalidValue;
}

}  // namespace tc
}  // namespace k
}  // namespace sn
