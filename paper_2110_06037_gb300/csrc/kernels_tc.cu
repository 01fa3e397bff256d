// Implicit-GEMM convolution on tcgen05 tensor cores (placeholder: no variants yet).
#include "kern_common.cuh"

namespace sn {
namespace k {

int32_t conv_tc_variants(const Layer &, const Shape &, sn_schema) { return 0; }
const char *conv_tc_variant_name(int32_t) { return "?"; }
cudaError_t conv_tc(const LaunchArgs &) { return cudaErrorNotSupported; }

}  // namespace k
}  // namespace sn
