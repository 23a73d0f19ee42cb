// ea_server_s.cu -- server kernels with the Adam moments at the server.
#include "ea_server.cuh"

namespace ea {
cudaError_t launch_server_s(const ServerArgs &a, cudaStream_t s) { return launch_server_mode<MODE_S>(a, s); }
}  // namespace ea
