// qs_step_128x128.cu -- write-back kernel instantiations for dk = 128, dv = 128.
#include "qs_step_impl.cuh"
#include "qs_wb_row.cuh"

namespace qs {
cudaError_t launch_step_128x128(const qstate_cfg& cfg, int src_packed, int dst_packed,
                            const StepParams& p, cudaStream_t stream) {
    return launch_step_shape<128, 128>(cfg, src_packed, dst_packed, p, stream);
}
cudaError_t launch_wb_row_128x128(const qstate_cfg& cfg, const StepParams& p, cudaStream_t stream) {
    return launch_wb_row_t<128, 128, 8>(cfg, p, stream);
}
cudaError_t launch_wb_chunk_128x128(const qstate_cfg& cfg, const StepParams& p, cudaStream_t stream) {
    return launch_wb_row_t<128, 128, 8, true>(cfg, p, stream);
}
}  // namespace qs
