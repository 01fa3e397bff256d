// Stream-K instantiations of the tensor-core convolution kernel (tc_conv.cuh),
// in a translation unit of their own so that they compile beside the others.
#include "tc_conv.cuh"

namespace sn {
namespace k {
namespace tc {

template <typename T, int BN, int KB>
static cudaError_t launch_sk_t(bool implicit, const CUtensorMap *mA, const CUtensorMap &mB, const CUtensorMap &mY,
                               const CUtensorMap &mR, const Params &p, cudaStream_t st) {
    return implicit ? launch<T, BN, true, 1, KB, false, 1, 1, true>(mA, mB, mY, mR, p, st)
                    : launch<T, BN, false, 1, KB, false, 1, 1, true>(mA, mB, mY, mR, p, st);
}

template <typename T>
static cudaError_t launch_sk_dt(int bn, int kb, bool implicit, const CUtensorMap *mA, const CUtensorMap &mB,
                                const CUtensorMap &mY, const CUtensorMap &mR, const Params &p, cudaStream_t st) {
    if (bn == 128 && kb == 1) return launch_sk_t<T, 128, 1>(implicit, mA, mB, mY, mR, p, st);
    if (bn == 128 && kb == 2) return launch_sk_t<T, 128, 2>(implicit, mA, mB, mY, mR, p, st);
    if (bn == 256 && kb == 1) return launch_sk_t<T, 256, 1>(implicit, mA, mB, mY, mR, p, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_sk(int dtype, int bn, int kb, bool implicit, const CUtensorMap *mA, const CUtensorMap &mB,
                      const CUtensorMap &mY, const CUtensorMap &mR, const Params &p, cudaStream_t st) {
    if (dtype == SN_BF16) return launch_sk_dt<__nv_bfloat16>(bn, kb, implicit, mA, mB, mY, mR, p, st);
    if (dtype == SN_F16) return launch_sk_dt<__half>(bn, kb, implicit, mA, mB, mY, mR, p, st);
    return cudaErrorInvalidValue;
}

}  // namespace tc
}  // namespace k
}  // namespace sn
