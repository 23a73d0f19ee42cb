// ea_server_w_q2.cu -- server kernels, Adam moments at the workers (the paper's Algorithm 1), uniform-grid broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_W, QK_UNIF>(const ServerArgs &, cudaStream_t);
template cudaError_t launch_server_grouped_for_qs<MODE_W, QK_UNIF>(const ServerArgs &, int, cudaStream_t);
template cudaError_t server_grouped_shape_for_qs<MODE_W, QK_UNIF>(int, GroupedShape *);
}  // namespace ea
