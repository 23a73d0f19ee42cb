// ea_server_w_q3.cu -- server kernels, Adam moments at the workers (the paper's Algorithm 1), power-of-two broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_W, QK_POW2>(const ServerArgs &, cudaStream_t);
}  // namespace ea
