// ea_server_w_q3.cu -- server kernels, Adam moments at the workers (the paper's Algorithm 1), power-of-two broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_W, QK_POW2>(const ServerArgs &, cudaStream_t);
template cudaError_t launch_server_grouped_for_qs<MODE_W, QK_POW2>(const ServerArgs &, int, cudaStream_t);
template cudaError_t server_grouped_shape_for_qs<MODE_W, QK_POW2>(int, GroupedShape *);
}  // namespace ea
