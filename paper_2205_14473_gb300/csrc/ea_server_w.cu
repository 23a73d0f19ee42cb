// ea_server_w.cu -- server kernels with the Adam moments at the workers (the paper's Algorithm 1).
#include "ea_server.cuh"

namespace ea {
cudaError_t launch_server_w(const ServerArgs &a, cudaStream_t s) { return launch_server_mode<MODE_W>(a, s); }
}  // namespace ea
