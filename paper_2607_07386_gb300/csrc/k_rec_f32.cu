// K-REC kernels for fp32 storage (see k_rec_impl.cuh).
#include "k_rec_impl.cuh"

namespace sdm {
cudaError_t launch_recur_f32(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s) {
    return launch_rec_dtype<F32>(p, a, hz, vec_lists, s);
}
}  // namespace sdm
