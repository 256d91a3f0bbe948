// cg_tc.h -- tensor-core (tcgen05) kernels of the row path: eligibility and launchers.
#pragma once

#include "cg_launch.h"

namespace cg {

bool tc_row_encode_eligible(const RowArgs& a);
bool tc_row_decode_eligible(const RowArgs& a);
cudaError_t tc_launch_row_encode(const RowArgs& a, cudaStream_t st);
cudaError_t tc_launch_row_decode(const RowArgs& a, cudaStream_t st);
bool tc_key_encode_eligible(const RowArgs& a);
cudaError_t tc_launch_key_encode(const RowArgs& a, cudaStream_t st);
bool tc_key_decode_eligible(const RowArgs& a);
cudaError_t tc_launch_key_decode(const RowArgs& a, cudaStream_t st);

}  // namespace cg
