// The commit step of a cycle (Sec. 2.4, "Update and Iterate"): the rows of a block of
// accepted positions are gathered into a dense batch; the runtime then runs Eq. 1 and the
// cascade over them (fe_runtime.cu), with one attention launch per row index so that a row
// reads the rows committed before it from the cache.
#include "fe_kernels.h"
#include "fe_common.cuh"

namespace fe {

// Row r = b * nb + j of the block (j = 0 .. nb - 1, row index i = i0 + j of sequence b):
// its feature row feat[b][i] (row_bytes bytes, 16-byte aligned) and its token; rows at or
// past n_rows[b] take token 0 (their outputs are computed but never stored).
__global__ void __launch_bounds__(128) commit_gather_kernel(const unsigned char* feat, const int* tok,
                                                            const int* n_rows, int L, int i0, int nb,
                                                            int row_bytes, unsigned char* cfeat, int* ctok) {
    const int r = blockIdx.x, b = r / nb, i = i0 + r % nb;
    const uint4* src = reinterpret_cast<const uint4*>(feat + ((size_t)b * L + i) * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>(cfeat + (size_t)r * row_bytes);
    for (int k = threadIdx.x; k < row_bytes / 16; k += blockDim.x) dst[k] = src[k];
    if (threadIdx.x == 0) ctok[r] = i < n_rows[b] ? tok[(size_t)b * L + i] : 0;
}

cudaError_t launch_commit_gather(const void* feat, const int* tok, const int* n_rows, int B, int L, int i0, int nb,
                                 int row_bytes, void* cfeat, int* ctok, cudaStream_t st) {
    if (B < 1 || nb < 1 || row_bytes % 16) return cudaErrorInvalidValue;
    commit_gather_kernel<<<B * nb, 128, 0, st>>>((const unsigned char*)feat, tok, n_rows, L, i0, nb, row_bytes,
                                                 (unsigned char*)cfeat, ctok);
    return cudaGetLastError();
}

}  // namespace fe
