// dar_backward_f32.cu -- the gradient kernels of dar_backward.cuh for fp32 storage.
#include "dar_backward.cuh"

namespace dar {
namespace bwd {

cudaError_t run_f32(int dd, const Args &a, cudaStream_t s) { return run_type<float>(dd, a, s); }

}  // namespace bwd
}  // namespace dar
