// common.cuh -- device helpers shared by the kernels of libmtp (sm_103a).
//
// Inline PTX for the Blackwell data movers used here: mbarrier
// (transaction-count barriers in shared memory), cp.async.bulk (the TMA
// engine's 1-D bulk copy global -> shared) and griddepcontrol (programmatic
// dependent launch).  Every wait is bounded: when it runs out the kernel sets
// the device error word instead of spinning forever.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mtp {

constexpr unsigned FULL_MASK = 0xffffffffu;

// bits of the device error word (ctx->d_err); the host maps any bit to MTP_ERR_DEVICE
enum DeviceError : int { ERR_WAIT_TIMEOUT = 1, ERR_BOUNDS = 2 };

// Bound on mbarrier polls: far above any legitimate copy latency (a few us),
// far below a hang.
constexpr uint32_t MBAR_MAX_POLLS = 1u << 20;

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// make an initialised mbarrier visible to the async (TMA) proxy
__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

// Bounded wait for phase `parity` of `bar`.  On time-out sets ERR_WAIT_TIMEOUT
// and returns false; callers then skip the work that needed the data.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* err) {
    for (uint32_t i = 0; i < MBAR_MAX_POLLS; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    if (err) atomicOr(err, ERR_WAIT_TIMEOUT);
    return false;
}

// Split cluster barrier: every thread of the cluster arrives, then waits.
// arrive.release makes this thread's earlier writes (shared memory included)
// visible to threads that return from their wait; arrive.relaxed orders
// nothing and only signals progress (e.g. "done reading peers' memory").
__device__ __forceinline__ void cluster_arrive_release() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Orders this thread's earlier generic-proxy accesses of shared memory (and
// those made visible to it by a barrier) before its later async-proxy copies.
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Shared-memory address of `p` (this CTA's shared memory) in the CTA of
// cluster rank `rank`, for ld.shared::cluster.
__device__ __forceinline__ uint32_t dsmem_addr(const void* p, int rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
    return r;
}
__device__ __forceinline__ float ld_dsmem(uint32_t addr) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr));
    return v;
}
__device__ __forceinline__ float2 ld_dsmem2(uint32_t addr) {  // 8-byte aligned
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
    return v;
}
__device__ __forceinline__ float4 ld_dsmem4(uint32_t addr) {  // 16-byte aligned
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr));
    return v;
}

// 1-D bulk copy global -> this CTA's shared memory, completing on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// An L2 access policy under which the lines an access touches are the first
// to be evicted.  Weights are streamed once per decode step (more bytes than
// L2 holds); copied under this policy they stop pushing out what the next
// kernels reuse from L2: code, activations, the cached keys and values, log Q.
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// bulk_copy_g2s with an L2 policy (l2_evict_first_policy for streamed weights).
__device__ __forceinline__ void bulk_copy_g2s_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                                   uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// Bulk prefetch of a global range into L2 (no destination, no completion).
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Programmatic dependent launch: wait until the preceding kernel in the stream
// has completed and its writes are visible (a no-op without the attribute).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Allow the next kernel in the stream to be scheduled (it still waits in pdl_wait).
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL_MASK, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(FULL_MASK, v, o));
    return v;
}

// bf16 <-> fp32 (bf16 -> fp32 is exact: the bf16 bits are the high half)
__device__ __forceinline__ float bf16_lo(uint32_t pair) { return __uint_as_float(pair << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t pair) { return __uint_as_float(pair & 0xffff0000u); }
__device__ __forceinline__ uint16_t f32_to_bf16_bits(float v) {
    __nv_bfloat16 b = __float2bfloat16_rn(v);
    return *reinterpret_cast<uint16_t*>(&b);
}

// four consecutive weights as fp32, from shared or global memory
__device__ __forceinline__ void load4(const __nv_bfloat16* p, float (&w)[4]) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    w[0] = bf16_lo(u.x); w[1] = bf16_hi(u.x); w[2] = bf16_lo(u.y); w[3] = bf16_hi(u.y);
}
__device__ __forceinline__ void load4(const float* p, float (&w)[4]) {
    const float4 u = *reinterpret_cast<const float4*>(p);
    w[0] = u.x; w[1] = u.y; w[2] = u.z; w[3] = u.w;
}

// ---- launch timeline (tracing option) --------------------------------------
// A traced launch owns TRACE_WORDS u64 words: earliest CTA start, latest CTA
// past the dependency wait, latest CTA end, then TRACE_MARKS phase marks
// (latest CTA past each mark), all from %globaltimer (ns).
constexpr int TRACE_MARKS = 8;
constexpr int TRACE_WORDS = 3 + TRACE_MARKS;

__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void trace_start(unsigned long long* tr) {
    if (tr && threadIdx.x == 0) atomicMin(tr, globaltimer());
}
__device__ __forceinline__ void trace_wait(unsigned long long* tr) {
    if (tr && threadIdx.x == 0) atomicMax(tr + 1, globaltimer());
}
__device__ __forceinline__ void trace_mark(unsigned long long* tr, int i) {
    if (tr && threadIdx.x == 0) atomicMax(tr + 3 + i, globaltimer());
}
struct TraceEnd {
    unsigned long long* tr;
    __device__ explicit TraceEnd(unsigned long long* t) : tr(t) { trace_start(t); }
    __device__ ~TraceEnd() {
        if (tr && threadIdx.x == 0) atomicMax(tr + 2, globaltimer());
    }
};

// Exact GELU, x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2)), with CUDA's erff.
__device__ __forceinline__ float gelu_erf(float x) { return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f)); }

}  // namespace mtp
