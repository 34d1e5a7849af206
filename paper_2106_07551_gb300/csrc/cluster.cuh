// Thread-block-cluster helpers: distributed shared memory (DSMEM) access to a
// peer CTA's shared memory and a cluster-wide synchronisation whose waits are
// bounded (epoch flags polled with a time limit, never an unbounded barrier).
#pragma once

#include <cstdint>

#include "device_common.cuh"

namespace malib {
namespace cl {

__device__ __forceinline__ uint32_t rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// shared::cluster address of `p` (this CTA's shared memory) in CTA `r`.
__device__ __forceinline__ uint32_t map(const void* p, uint32_t r) {
    uint32_t out;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(out) : "r"(smem_u32(p)), "r"(r));
    return out;
}

__device__ __forceinline__ void st_u32(uint32_t addr, uint32_t v) {
    asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ void st_f32(uint32_t addr, float v) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void st_v4(uint32_t addr, uint4 v) {
    asm volatile("st.shared::cluster.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x),
                 "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint32_t ld_u32(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t atomic_add(uint32_t addr, uint32_t v) {
    uint32_t old;
    asm volatile("atom.relaxed.cluster.shared::cluster.add.u32 %0, [%1], %2;"
                 : "=r"(old)
                 : "r"(addr), "r"(v)
                 : "memory");
    return old;
}

// Asynchronous 16-byte store into a peer CTA's shared memory that, once the
// data is written, completes 16 bytes of transaction count on the mbarrier at
// `remote_bar` (both addresses from map(), in the same peer CTA).
__device__ __forceinline__ void st_async_v4(uint32_t remote_addr, uint4 v, uint32_t remote_bar) {
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, "
        "[%5];" ::"r"(remote_addr),
        "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(remote_bar)
        : "memory");
}

// One attempt at the phase `parity` of a local mbarrier whose transactions come
// from peer CTAs (acquire at cluster scope); true when it has completed.
__device__ __forceinline__ bool try_wait_cluster(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n"
        " mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait (at most limit_ns) for the phase `parity` of a local mbarrier
// whose transactions come from peer CTAs; acquires at cluster scope so the
// peers' completed stores are visible. Returns false on expiry.
__device__ __forceinline__ bool wait_cluster_bounded(uint64_t* bar, uint32_t parity,
                                                     uint64_t limit_ns) {
    auto try_once = [&]() {
        uint32_t ok;
        asm volatile(
            "{\n .reg .pred p;\n"
            " mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
            " selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(smem_u32(bar)), "r"(parity)
            : "memory");
        return ok != 0;
    };
    if (try_once()) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (try_once()) return true;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

__device__ __forceinline__ void fence_cluster() {
    asm volatile("fence.acq_rel.cluster;" ::: "memory");
}

// Cluster-wide synchronisation. Every thread of every CTA of the cluster calls
// it with the same epoch (increasing). flags: this CTA's array of `size`
// epoch slots (one per source CTA), zero-initialised and never reset. The CTA
// synchronises (so the signalling threads have observed every write of the
// CTA), then thread r releases the epoch into slot [my rank] of CTA r at
// cluster scope; thread 0 then polls
// its own slots until every source has reached the epoch, for at most
// kWaitLimitNs. Returns false (and raises ERRBIT_TIMEOUT) on expiry; callers
// keep executing the same sequence of syncs so that no CTA of the cluster is
// left waiting.
__device__ __forceinline__ bool sync(uint32_t* flags, uint32_t epoch, uint32_t size, uint32_t me,
                                     int* err, uint32_t* ok_slot) {
    __syncthreads();
    if (threadIdx.x < size) {
        const uint32_t a = map(&flags[me], threadIdx.x);
        asm volatile("st.release.cluster.shared::cluster.u32 [%0], %1;" ::"r"(a), "r"(epoch)
                     : "memory");
    }
    if (threadIdx.x == 0) {
        bool ok = true;
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t r = 0; r < size && ok; ++r) {
            for (uint32_t spin = 0;; ++spin) {
                uint32_t v;
                asm volatile("ld.acquire.cluster.shared::cta.u32 %0, [%1];"
                             : "=r"(v)
                             : "r"(smem_u32(&flags[r]))
                             : "memory");
                if ((int32_t)(v - epoch) >= 0) break;
                if ((spin & 63u) == 63u && globaltimer_ns() - t0 > kWaitLimitNs) { ok = false; break; }
            }
        }
        if (!ok) atomicOr(err, ERRBIT_TIMEOUT);
        *ok_slot = ok ? 1u : 0u;
    }
    __syncthreads();
    return *ok_slot != 0;
}

}  // namespace cl
}  // namespace malib
