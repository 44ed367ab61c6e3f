#include "tc_path.h"

namespace jpi {

bool tc_supported(const jpi_handle*) { return false; }
jpi_status tc_pack_layers(jpi_handle*, const jpi_weights*, float*, bool) { return JPI_ERR_UNSUPPORTED; }
jpi_status tc_prepare(jpi_handle*) { return JPI_OK; }
jpi_status tc_launch_layer(jpi_handle*, int, int, int, int, cudaStream_t) { return JPI_ERR_UNSUPPORTED; }
jpi_status tc_launch_op(jpi_handle*, int, int, int, int, int, cudaStream_t) { return JPI_ERR_UNSUPPORTED; }
void tc_release(jpi_handle*) {}

}  // namespace jpi
