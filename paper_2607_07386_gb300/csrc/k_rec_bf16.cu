// K-REC kernels for bfloat16 storage (see k_rec_impl.cuh).
#include "k_rec_impl.cuh"

namespace sdm {
cudaError_t launch_recur_bf16(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s) {
    return launch_rec_dtype<BF16>(p, a, hz, vec_lists, s);
}
}  // namespace sdm
