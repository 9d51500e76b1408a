// Internal helpers shared by the sm_103a kernels of the PLD+ library.
#pragma once

#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pldp.h"

namespace pldp {

namespace cg = cooperative_groups;

// ---------------------------------------------------------------------------
// host-side error reporting (defined in abi.cu)
// ---------------------------------------------------------------------------
pldp_status fail(pldp_status code, const char* fmt, ...);
pldp_status check_launch(const char* what);
int sm_count();  // SMs of the current device
// CTAs of `kernel` that fit on the whole current device at once (cached).
int resident_blocks(const void* kernel, int threads, size_t smem);

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ---------------------------------------------------------------------------
// element loads
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// Order-preserving map of a float onto uint32 (larger float -> larger key).
// -0.0 is folded onto +0.0 first, so equal values give equal keys.
__device__ __forceinline__ uint32_t ordered_key(float v) {
    uint32_t u = __float_as_uint(v == 0.0f ? 0.0f : v);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Packed (value, index) key: the larger value wins, ties go to the smaller index.
__device__ __forceinline__ unsigned long long pack_key(float v, uint32_t idx) {
    return (static_cast<unsigned long long>(ordered_key(v)) << 32) |
           static_cast<unsigned long long>(0xFFFFFFFFu - idx);
}
__device__ __forceinline__ uint32_t key_index(unsigned long long k) {
    return 0xFFFFFFFFu - static_cast<uint32_t>(k & 0xFFFFFFFFull);
}
__device__ __forceinline__ float key_value(unsigned long long k) {
    uint32_t o = static_cast<uint32_t>(k >> 32);
    uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
    return __uint_as_float(u);
}

__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        unsigned long long w = __shfl_xor_sync(0xFFFFFFFFu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

// Max and first index of the max of one 16-byte vector (8 bf16 or 4 fp32): a
// packed max first, the index search only when the caller needs it.
__device__ __forceinline__ float vmax(const uint4& x, __nv_bfloat16) {
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&x.x);
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&x.y);
    const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&x.z);
    const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&x.w);
    const __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
    return fmaxf(__low2float(m), __high2float(m));
}
__device__ __forceinline__ int vfirst(const uint4& x, float m, __nv_bfloat16) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (__uint_as_float(w[k] << 16) == m) return 2 * k;
        if (__uint_as_float(w[k] & 0xFFFF0000u) == m) return 2 * k + 1;
    }
    return 0;
}
__device__ __forceinline__ float vmax(const uint4& x, float) {
    return fmaxf(fmaxf(__uint_as_float(x.x), __uint_as_float(x.y)),
                 fmaxf(__uint_as_float(x.z), __uint_as_float(x.w)));
}
__device__ __forceinline__ int vfirst(const uint4& x, float m, float) {
    if (__uint_as_float(x.x) == m) return 0;
    if (__uint_as_float(x.y) == m) return 1;
    if (__uint_as_float(x.z) == m) return 2;
    return 3;
}

// Streaming 16-byte global load (read-once data: no L1 allocation).
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// ---------------------------------------------------------------------------
// mbarrier + bulk async copy (global -> this CTA's shared memory)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

// One bulk copy of `bytes` (multiple of 16; both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_g2s(void* dst_smem, const void* src_gmem, uint32_t bytes,
                                         uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_u32(dst_smem)), "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// Bounded wait on phase `parity` of an mbarrier.  Returns false if the phase did
// not complete within `max_polls` polls (the caller records a timeout).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t max_polls) {
    uint32_t done = 0;
    for (uint32_t i = 0; i < max_polls; ++i) {
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(smem_u32(bar)), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

constexpr uint32_t kMbarPolls = 1u << 22;   // each try_wait may suspend; ~tens of ms bound

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  Kernels of a step are launched so that the
// next one may be scheduled while the previous one runs; every kernel first
// waits for the grids it depends on to finish (and their writes to be visible),
// then lets its own dependent be scheduled.  Without the launch attribute both
// instructions are no-ops.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_enter() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The wait alone: the next kernel is then scheduled only as this grid's CTAs
// finish, for a kernel whose dependent is heavy enough (registers, threads) to
// crowd out this grid's last CTAs if it were resident early.
__device__ __forceinline__ void pdl_wait_only() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Launches `kernel` with programmatic stream serialisation (and an optional
// cluster shape, cluster_x > 0).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       int cluster_x, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    int n = 0;
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
    if (cluster_x > 0) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = cluster_x;
        attr[n].val.clusterDim.y = 1;
        attr[n].val.clusterDim.z = 1;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

}  // namespace pldp
