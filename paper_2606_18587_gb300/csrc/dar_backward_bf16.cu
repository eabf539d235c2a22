// dar_backward_bf16.cu -- the gradient kernels of dar_backward.cuh for bf16 storage.
#include "dar_backward.cuh"

namespace dar {
namespace bwd {

cudaError_t run_bf16(int dd, const Args &a, cudaStream_t s) { return run_type<bf16>(dd, a, s); }

}  // namespace bwd
}  // namespace dar
