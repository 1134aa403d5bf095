// Self-check of the tensor-core operand layouts: one 128 x 128 x 128 bf16 product on tcgen05
// with TMEM accumulation, operands loaded by TMA (128-byte swizzle) or written by threads in
// the same swizzled layout, in each combination of K-major / MN-major A and B that the chunk
// kernels use.  D = op(X) op(Y) with op(X) = X (K-major) or X^T (MN-major), op(Y) = Y^T
// (K-major) or Y (MN-major), for X, Y row-major [128 x 128] bf16.
#include "../../include/cyfa.h"
#include "kernels.h"
#include "tc_common.cuh"

namespace cyfa {
namespace {

static __device__ int g_selftest_err;

__global__ void __launch_bounds__(128) selftest_kernel(const __grid_constant__ CUtensorMap mx,
                                                       const __grid_constant__ CUtensorMap my,
                                                       const __nv_bfloat16* X,
                                                       const __nv_bfloat16* Y, float* D,
                                                       int variant) {
    using namespace tc;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sX = smem;
    uint8_t* sY = smem + 32768;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 65536);
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 65536 + 64);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int a_mn = variant & 1, b_mn = (variant >> 1) & 1, by_threads = (variant >> 2) & 1;

    if (tid == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(s_taddr, 128);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    bool ok = true;

    if (by_threads) {
        for (int e = tid; e < 128 * 128; e += 128) {
            const int r = e >> 7, c = e & 127;
            *reinterpret_cast<__nv_bfloat16*>(sX + swz_off(r, c, 128)) = X[e];
            *reinterpret_cast<__nv_bfloat16*>(sY + swz_off(r, c, 128)) = Y[e];
        }
        fence_async_smem();
        __syncthreads();
    } else {
        if (tid == 0) {
            mbar_expect_tx(&bars[0], 65536);
            tma_load_2d(sX, &mx, 0, 0, &bars[0]);
            tma_load_2d(sX + 16384, &mx, 64, 0, &bars[0]);
            tma_load_2d(sY, &my, 0, 0, &bars[0]);
            tma_load_2d(sY + 16384, &my, 64, 0, &bars[0]);
        }
        ok = mbar_wait(&bars[0], 0);
    }
    if (ok && tid == 0) {
        const uint32_t bx = smem_u32(sX), byy = smem_u32(sY);
        const uint32_t idesc = idesc_bf16(128, 128, a_mn, b_mn);
        for (int k = 0; k < 8; ++k) {
            const uint64_t ad = a_mn ? mnmajor_desc(bx, 128, k) : kmajor_desc(bx, 128, k);
            const uint64_t bd = b_mn ? mnmajor_desc(byy, 128, k) : kmajor_desc(byy, 128, k);
            mma_bf16(taddr, ad, bd, idesc, k > 0);
        }
        mma_commit(&bars[1]);
    }
    if (ok) ok = mbar_wait(&bars[1], 0);
    tc_fence_after();
    if (ok) {
        const int row = warp * 32 + lane;
        for (int c0 = 0; c0 < 128; c0 += 32) {
            float v[32];
            tmem_ld32(taddr + ((uint32_t)(warp * 32) << 16) + c0, v);
            for (int i = 0; i < 32; ++i) D[row * 128 + c0 + i] = v[i];
        }
    } else if (lane == 0) {
        atomicExch(&g_selftest_err, 1);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, 128);
}

// Expiry of a bounded wait: one thread waits on an mbarrier that nothing ever arrives on, with
// the kernels' own wait (mbar_wait_for) given a limit of `limit_us`; when it gives up, the error
// word is set and the kernel returns normally (no trap, no fault: the context stays usable).
static __device__ int g_timeout_err;

__global__ void timeout_probe_kernel(uint32_t limit_us, unsigned long long* elapsed_ns) {
    using namespace tc;
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
        const unsigned long long t0 = globaltimer_ns();
        const bool done = mbar_wait_for(&bar, 0, 1000ull * limit_us);
        if (elapsed_ns) *elapsed_ns = globaltimer_ns() - t0;
        if (!done) atomicExch(&g_timeout_err, CYFA_ERR_TIMEOUT);
    }
}

}  // namespace

cudaError_t launch_timeout_probe(unsigned limit_us, unsigned long long* elapsed_ns,
                                 cudaStream_t st, int* host_err) {
    int zero = 0;
    cudaError_t e = cudaMemcpyToSymbolAsync(g_timeout_err, &zero, sizeof(int), 0,
                                            cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return e;
    {
        LaunchScope ls_("selftest_timeout", st);
        timeout_probe_kernel<<<1, 32, 0, st>>>(limit_us, elapsed_ns);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbolAsync(host_err, g_timeout_err, sizeof(int), 0, cudaMemcpyDeviceToHost,
                                  st);
    if (e != cudaSuccess) return e;
    return cudaStreamSynchronize(st);
}

cudaError_t launch_selftest_mma(int variant, const void* X, const void* Y, float* D,
                                cudaStream_t st, int* host_err) {
    CUtensorMap mx, my;
    const unsigned long long dims[2] = {128, 128}, strides[1] = {256};
    const unsigned box[2] = {64, 128};
    if (!make_tmap_bf16(&mx, X, 2, dims, strides, box) ||
        !make_tmap_bf16(&my, Y, 2, dims, strides, box))
        return cudaErrorInvalidValue;
    int zero = 0;
    cudaError_t e = cudaMemcpyToSymbolAsync(g_selftest_err, &zero, sizeof(int), 0,
                                            cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return e;
    const int smem = 65536 + 1024 + 128;
    cudaFuncSetAttribute(selftest_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    {
        LaunchScope ls_("selftest_mma", st);
        selftest_kernel<<<1, 128, smem, st>>>(mx, my, static_cast<const __nv_bfloat16*>(X),
                                              static_cast<const __nv_bfloat16*>(Y), D, variant);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbolAsync(host_err, g_selftest_err, sizeof(int), 0,
                                  cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    return cudaStreamSynchronize(st);
}

}  // namespace cyfa

extern "C" int cyfa_selftest_mma(int variant, const void* X, const void* Y, float* D,
                                 void* stream) {
    if (variant < 0 || variant > 7 || !X || !Y || !D) return CYFA_ERR_ARG;
    int err = 0;
    const cudaError_t e =
        cyfa::launch_selftest_mma(variant, X, Y, D, static_cast<cudaStream_t>(stream), &err);
    if (e != cudaSuccess) return CYFA_ERR_CUDA;
    return err ? CYFA_ERR_TIMEOUT : CYFA_OK;
}

extern "C" int cyfa_selftest_timeout(unsigned int limit_us, unsigned long long* elapsed_ns,
                                     void* stream) {
    if (limit_us == 0 || limit_us > 1000000u) return CYFA_ERR_ARG;
    int err = 0;
    const cudaError_t e =
        cyfa::launch_timeout_probe(limit_us, elapsed_ns, static_cast<cudaStream_t>(stream), &err);
    if (e != cudaSuccess) return CYFA_ERR_CUDA;
    return err ? CYFA_ERR_TIMEOUT : CYFA_OK;
}
