// decoder_kernel_gelu.cu -- instantiations of the decoder kernel with the GELU feed-forward
// activation, AAP linears (Sec. 4.1).
#include "decoder_kernel.cuh"

namespace aecct {

template cudaError_t launch_decode<32, 0, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, 0, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 0, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<32, 1, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, 1, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 1, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 2, 1, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t prepare_decode_kernel<32, 0, 1, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<64, 0, 1, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 0, 1, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<32, 1, 1, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<64, 1, 1, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 1, 1, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 2, 1, 0>(int, uint32_t, int *);

}  // namespace aecct
