// Checks of the bounds-checked debug build (TFG_CHECK_BOUNDS=1): api.cu runs
// them before every launch that takes caller-built index arrays or buffers,
// so a bad index or a too-small buffer is reported as an error code and no
// kernel ever reads out of bounds.  Not a step of the paper's method; the
// default build compiles these helpers but never calls them.
//
//   allocation_range  [base, base + size) of the device allocation holding a
//                     pointer (the driver's cuMemGetAddressRange, looked up
//                     through the runtime, so the library links no libcuda)
//   csr_ends          rowptr[0] and rowptr[n], copied to the host
//   validate_csr      rowptr non-decreasing (when given), every col id in
//                     [0, n) and every perm id in [0, E) (each when given):
//                     one grid-stride pass, flags ORed
#include <cuda.h>

#include <mutex>

#include "common.cuh"

namespace tfg {
namespace {

__device__ int g_check_flags;

constexpr int kRowFlag = 1, kColFlag = 2, kPermFlag = 4;

// rows = n with a rowptr, 0 without; ids are checked against [0, n)
__global__ void validate_csr_kernel(const int32_t *__restrict__ rowptr,
                                    const int32_t *__restrict__ col,
                                    const int32_t *__restrict__ perm, int64_t rows, int64_t e,
                                    int64_t n) {
    int flags = 0;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < rows + e;
         i += stride) {
        if (i < rows) {
            if (rowptr[i] > rowptr[i + 1]) flags |= kRowFlag;
        } else {
            const int64_t k = i - rows;
            if (col) {
                const int32_t c = col[k];
                if (c < 0 || c >= n) flags |= kColFlag;
            }
            if (perm) {
                const int32_t p = perm[k];
                if (p < 0 || p >= e) flags |= kPermFlag;
            }
        }
    }
    if (flags) atomicOr(&g_check_flags, flags);
}

using AddressRangeFn = CUresult (*)(CUdeviceptr *, size_t *, CUdeviceptr);

AddressRangeFn address_range_fn() {
    static std::once_flag once;
    static AddressRangeFn fn = nullptr;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuMemGetAddressRange", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<AddressRangeFn>(f);
    });
    return fn;
}

}  // namespace

bool allocation_range(const void *p, uintptr_t *base, size_t *size) {
    const AddressRangeFn fn = address_range_fn();
    if (fn == nullptr || p == nullptr) return false;
    CUdeviceptr b = 0;
    size_t s = 0;
    if (fn(&b, &s, reinterpret_cast<CUdeviceptr>(p)) != CUDA_SUCCESS) return false;
    *base = static_cast<uintptr_t>(b);
    *size = s;
    return true;
}

cudaError_t csr_ends(const int32_t *rowptr, int64_t n, int32_t *first, int32_t *last,
                     cudaStream_t s) {
    cudaError_t err = cudaMemcpyAsync(first, rowptr, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (err == cudaSuccess)
        err = cudaMemcpyAsync(last, rowptr + n, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (err == cudaSuccess) err = cudaStreamSynchronize(s);
    return err;
}

cudaError_t validate_csr(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                         int64_t n, int64_t e, int *flags, cudaStream_t s) {
    const int zero = 0;
    cudaError_t err = cudaMemcpyToSymbolAsync(g_check_flags, &zero, sizeof(int), 0,
                                              cudaMemcpyHostToDevice, s);
    if (err != cudaSuccess) return err;
    const int64_t rows = rowptr ? n : 0;               // no rowptr: the ids alone
    const int64_t ids = (col || perm) ? e : 0;         // neither given: no id to read
    if (rows + ids > 0) {
        const int grid = static_cast<int>(min64(ceil_div(rows + ids, 256), int64_t(sm_count()) * 8));
        validate_csr_kernel<<<grid, 256, 0, s>>>(rowptr, col, perm, rows, ids, n);
        err = cudaGetLastError();
        if (err != cudaSuccess) return err;
    }
    err = cudaMemcpyFromSymbolAsync(flags, g_check_flags, sizeof(int), 0, cudaMemcpyDeviceToHost, s);
    if (err == cudaSuccess) err = cudaStreamSynchronize(s);
    return err;
}

}  // namespace tfg
