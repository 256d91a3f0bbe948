// cg_tc.cu -- tensor-core (tcgen05) kernels of the row path.
#include "cg_tc.h"

namespace cg {

bool tc_row_encode_eligible(const RowArgs&) { return false; }
bool tc_row_decode_eligible(const RowArgs&) { return false; }
cudaError_t tc_launch_row_encode(const RowArgs&, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t tc_launch_row_decode(const RowArgs&, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace cg
