// ea_server_s_q0.cu -- server kernels, Adam moments at the server, identity broadcast.
#include "ea_server.cuh"

namespace ea {
template cudaError_t launch_server_for_qs<MODE_S, QK_IDENT>(const ServerArgs &, cudaStream_t);
template cudaError_t launch_server_grouped_for_qs<MODE_S, QK_IDENT>(const ServerArgs &, int, cudaStream_t);
template cudaError_t server_grouped_shape_for_qs<MODE_S, QK_IDENT>(int, GroupedShape *);
}  // namespace ea
