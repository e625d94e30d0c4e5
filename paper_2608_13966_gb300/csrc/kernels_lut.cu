// Instantiation of the Rubin INT3 lookup-table kernel (batches of up to
// kMaxBatch tensors; one tensor is a batch of one).
#include "recon_lut.cuh"

namespace quasar {

const void* lut_kernel() { return reinterpret_cast<const void*>(&k_recon_lut<kMaxBatch>); }

}  // namespace quasar
