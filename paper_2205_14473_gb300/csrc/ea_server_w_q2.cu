// ea_server_w_q2.cu -- server kernels, Adam moments at the workers (the paper's Algorithm 1), uniform-grid broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_W, QK_UNIF>(const ServerArgs &, cudaStream_t);
}  // namespace ea
