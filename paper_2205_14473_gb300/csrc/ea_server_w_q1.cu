// ea_server_w_q1.cu -- server kernels, Adam moments at the workers (the paper's Algorithm 1), scaled-sign broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_W, QK_SIGN>(const ServerArgs &, cudaStream_t);
template cudaError_t launch_server_lazy<MODE_W>(const ServerArgs &, bool, cudaStream_t);
}  // namespace ea
