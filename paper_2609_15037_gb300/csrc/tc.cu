// Tensor-core path of the step (placeholder until the tcgen05 kernels land).
#include <string>

#include "tc.h"

namespace moara {

struct TcState {
    int device;
    int* d_status;
    std::string err;
};

bool tc_supported(int, int, int, int, int, int) { return false; }

TcState* tc_create(int device, int* d_status) { return new TcState{device, d_status, {}}; }

void tc_destroy(TcState* st) { delete st; }

int tc_register(TcState*, int, const ModDev&, const moara_hparams&) { return MOARA_OK; }

int tc_step(TcState* st, const moara_hparams&, int, const int*, const void* const*, float, float, float,
            cudaStream_t, int64_t*, const TcProfile&) {
    st->err = "tensor-core path not available";
    return MOARA_ERR_UNSUPPORTED;
}

const char* tc_last_error(const TcState* st) { return st->err.c_str(); }

}  // namespace moara
