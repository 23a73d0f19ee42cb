// ea_server_s_q1.cu -- server kernels, Adam moments at the server, scaled-sign broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_S, QK_SIGN>(const ServerArgs &, cudaStream_t);
template cudaError_t launch_server_lazy<MODE_S>(const ServerArgs &, bool, cudaStream_t);
}  // namespace ea
