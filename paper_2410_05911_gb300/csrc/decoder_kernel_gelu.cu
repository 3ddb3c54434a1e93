// decoder_kernel_gelu.cu -- instantiations of the decoder kernel with the GELU feed-forward
// activation, AAP linears (Sec. 4.1).
#include "decoder_kernel.cuh"

namespace aecct {

template cudaError_t launch_decode<32, false, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, false, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, false, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<32, true, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, true, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, true, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t prepare_decode_kernel<32, false, 1, 0>(int, int *);
template cudaError_t prepare_decode_kernel<64, false, 1, 0>(int, int *);
template cudaError_t prepare_decode_kernel<128, false, 1, 0>(int, int *);
template cudaError_t prepare_decode_kernel<32, true, 1, 0>(int, int *);
template cudaError_t prepare_decode_kernel<64, true, 1, 0>(int, int *);
template cudaError_t prepare_decode_kernel<128, true, 1, 0>(int, int *);

}  // namespace aecct
