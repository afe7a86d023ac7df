// Device-side building blocks for the TaskPress kernels on sm_103a:
// mbarriers with bounded waits, TMA tile loads, tcgen05 (TMEM allocation,
// MMA issue/commit, TMEM loads) and shared-memory matrix descriptors.
//
// All PTX here is written from the public PTX ISA description of these
// instructions; no library headers beyond the CUDA runtime are used.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "tp_internal.h"

namespace tp {

// ---------------------------------------------------------------------------
// Small helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// 2^x on the special-function unit (PTX ex2.approx.ftz.f32).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Programmatic dependent launch: a kernel launched as a dependent may start
// while its predecessor in the stream finishes; grid_dep_wait() returns once
// the predecessor has completed and its writes are visible (at once when the
// kernel was not launched as a dependent).  grid_dep_launch() lets this
// kernel's own dependent be scheduled as soon as every CTA of this grid has
// issued it.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;"); }

// Records a device-side failure in the workspace status word (first writer wins).
__device__ __forceinline__ void set_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking test of the phase with parity `parity` (never suspends the
// thread; for event loops that poll several barriers).
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase of `bar` with parity `parity` to complete.  Gives up
// after kWaitLimitNs of wall time or as soon as another thread of the CTA
// raised `abort_flag`; returns false then (the caller unwinds).
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s

__device__ __forceinline__ bool mbar_wait_limit(uint64_t* bar, uint32_t parity,
                                                volatile int* abort_flag, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63) == 0) {
      if (*abort_flag) return false;
      if (global_timer_ns() - t0 > limit_ns) {
        *abort_flag = 1;
        return false;
      }
    }
  }
}

__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity,
                                          volatile int* abort_flag) {
  return mbar_wait_limit(bar, parity, abort_flag, kWaitLimitNs);
}

// ---------------------------------------------------------------------------
// Thread-block clusters: addresses in a peer CTA's shared memory, remote
// stores and mbarrier arrivals, and cluster-scope waits.
// ---------------------------------------------------------------------------
// Address of `local` (a shared-memory object of this CTA) in cluster CTA `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void* local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank));
  return r;
}

__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}

// Arrival (release at cluster scope) on an mbarrier of another cluster CTA.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(addr)
               : "memory");
}

// Arrival on an mbarrier of another cluster CTA with the default CTA-scope
// release: enough where the arrival only reports that this thread's own
// tensor-memory loads have completed (tcgen05.wait::ld), not data it wrote.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(addr) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// mbar_wait for a barrier whose arrivals come from other cluster CTAs (their
// writes before arriving are visible after it returns true).
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity,
                                                  volatile int* abort_flag) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((i & 63) == 0) {
      if (*abort_flag) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        return false;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// TMA (cp.async.bulk.tensor) - 3-D tiled load into shared memory, completion
// signalled on an mbarrier as transaction bytes.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_3d(void* smem_dst, const CUtensorMap* map, int x, int y,
                                            int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

// The same load with an L2 eviction-priority policy (createpolicy): the K and V
// streams, read once, take evict_first so that they do not push the freshly
// written scales and key scores, which the selection reads next, out of L2.
__device__ __forceinline__ void tma_load_3d_hint(void* smem_dst, const CUtensorMap* map, int x, int y,
                                                 int z, uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t policy;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
  return policy;
}

// 4-byte asynchronous global -> shared copy (no register staging); with
// valid == false nothing is read and the destination word is zero-filled.
__device__ __forceinline__ void cp_async4(void* smem_dst, const void* gsrc, bool valid) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(smem_u32(smem_dst)), "l"(gsrc),
               "r"(valid ? 4 : 0)
               : "memory");
}
// 16-byte asynchronous global -> shared copy (both addresses 16-byte aligned).
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc)
               : "memory");
}
// Waits for every cp.async this thread has issued.
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
// Closes this thread's current group of cp.async copies.
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
// Waits until at most N of this thread's committed groups are still in flight.
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Orders this thread's earlier generic-proxy shared-memory accesses before
// later async-proxy ones (a TMA write into a buffer that was just read).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05: tensor memory, MMA and loads (one CTA, cta_group::1)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulation.
__device__ __forceinline__ void mma_bf16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives once on `bar` when every tcgen05 op this thread issued so far completes.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// Instruction descriptor for kind::f16: bf16 A and B (both K-major), fp32 D,
// shape M x N (M in {64,128}; N a multiple of 16 up to 256).
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int m, int n) {
  return (1u << 4)                               // D format: f32
         | (1u << 7)                             // A format: bf16
         | (1u << 10)                            // B format: bf16
         | (static_cast<uint32_t>(n >> 3) << 17)  // N / 8
         | (static_cast<uint32_t>(m >> 4) << 24); // M / 16
}

// Shared-memory matrix descriptor of a K-major operand stored as 8-row x
// 128-byte swizzle atoms (128B swizzle; 1024 bytes between 8-row groups).
// `addr` is the shared-memory byte address of the first 16-element K slice.
__device__ __forceinline__ uint64_t sdesc_k128(uint32_t addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr & 0x3FFFFu) >> 4);  // start address
  d |= static_cast<uint64_t>(1) << 16;                 // leading byte offset (unused here)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;         // stride byte offset
  d |= static_cast<uint64_t>(1) << 46;                 // descriptor version
  d |= static_cast<uint64_t>(2) << 61;                 // 128-byte swizzle
  return d;
}

// Descriptor of a K-major bf16 operand with 32-byte rows (one K=16 step) in the
// 32-byte swizzle: 8-row atoms of 256 bytes; within an atom, 16-byte chunk c of
// row r sits at chunk position c ^ ((r >> 2) & 1).
__device__ __forceinline__ uint64_t sdesc_k32(uint32_t addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr & 0x3FFFFu) >> 4);  // start address
  d |= static_cast<uint64_t>(1) << 16;                 // leading byte offset (unused here)
  d |= static_cast<uint64_t>(256 >> 4) << 32;          // stride byte offset: 8 rows x 32 B
  d |= static_cast<uint64_t>(1) << 46;                 // descriptor version
  d |= static_cast<uint64_t>(6) << 61;                 // 32-byte swizzle
  return d;
}

// bf16 bits of x rounded to nearest, ties to even (finite x).
__device__ __forceinline__ uint32_t bf16_bits_rn(float x) {
  const uint32_t u = __float_as_uint(x);
  return (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
}

// Issues a load of 32 consecutive TMEM columns of this warp's 32 lanes (one
// lane per thread) without waiting; the registers become valid at the next
// tmem_wait() that names them.
__device__ __forceinline__ void tmem_ld32_async(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

// Waits for this thread's outstanding TMEM loads.  The registers of the load
// being completed are listed as read-write operands, so the compiler neither
// reads them before this point nor reuses them in between.
__device__ __forceinline__ void tmem_wait(uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;\n"
      : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
        "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
        "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]),
        "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]),
        "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
      :
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]^T: A (M = 128 rows on lanes, K packed two
// bf16 per 32-bit column) read from tensor memory, B from shared memory.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Stores 32 (x32) or 64 (x64) consecutive 32-bit columns of this warp's 32
// TMEM lanes from registers, then waits for the stores to complete.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};\n\t"
      "tcgen05.wait::st.sync.aligned;\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05 on a CTA pair (cta_group::2): the two CTAs of a cluster whose ranks
// differ only in bit 0 (scheduled on the two SMs of one TPC) share each MMA.
// A is split along M (each CTA supplies its 128 rows from its own shared
// memory), B along N (each CTA supplies N/2 rows, the even CTA the first
// half), both at the same shared-memory offsets in the two CTAs; each CTA's
// tensor memory receives its 128 rows of D with all N columns.  Allocation
// and release are collective: one warp of EACH CTA executes them with the
// same column count, and both receive the same address.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Every thread of every CTA of the cluster (release/acquire at cluster scope).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

__device__ __forceinline__ void tmem_alloc_pair(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// D (+)= A * B^T over the pair (M = 256 in the instruction descriptor),
// issued by one thread of the even CTA.
__device__ __forceinline__ void mma_bf16_ss_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                 uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives once on the mbarrier at `bar`'s offset in BOTH CTAs of the pair when
// every tcgen05 op this thread issued so far completes.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
  const uint16_t mask = 3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(mask)
      : "memory");
}

// Packed fp32 pairs (one instruction for two lanes of arithmetic).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// 32 consecutive TMEM columns of this warp's 32 lanes (one lane per thread),
// followed by the wait that makes the registers valid.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

// Radix key of a combined score: scores are non-negative fp32, so their bit
// patterns order like their values once -0, NaN and negatives map to +0.
__device__ __forceinline__ uint32_t score_key(float s) {
  return (s > 0.f) ? __float_as_uint(s) : 0u;
}

// Stages global floats src[ga, gb) into dst[g - g_ref] (g_ref a multiple of 4,
// dst 16-byte aligned): 16-byte cp.async over the aligned middle, 4-byte ones
// at the two ragged ends.  Called by every thread of the block.
__device__ __forceinline__ void stage_floats(float* dst, const float* src, int64_t ga, int64_t gb,
                                             int64_t g_ref) {
  if (gb <= ga) return;
  const int64_t a4 = (ga + 3) & ~int64_t(3), b4 = gb & ~int64_t(3);
  // a caller's array need only be 4-byte aligned: then every copy is 4 bytes
  if (a4 >= b4 || (reinterpret_cast<uintptr_t>(src) & 15) != 0) {
    for (int64_t g = ga + threadIdx.x; g < gb; g += blockDim.x) cp_async4(dst + (g - g_ref), src + g, true);
    return;
  }
  const int64_t groups = (b4 - a4) >> 2;
  for (int64_t q = threadIdx.x; q < groups; q += blockDim.x) {
    const int64_t g = a4 + 4 * q;
    cp_async16(dst + (g - g_ref), src + g);
  }
  const int head = static_cast<int>(a4 - ga), tail = static_cast<int>(gb - b4);
  if (static_cast<int>(threadIdx.x) < head) {
    const int64_t g = ga + threadIdx.x;
    cp_async4(dst + (g - g_ref), src + g, true);
  } else if (static_cast<int>(threadIdx.x) >= 32 && static_cast<int>(threadIdx.x) < 32 + tail) {
    const int64_t g = b4 + (threadIdx.x - 32);
    cp_async4(dst + (g - g_ref), src + g, true);
  }
}

// ---------------------------------------------------------------------------
// Block-wide helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ int warp_incl_scan(int v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  return v;
}

// Exclusive scan over the block (blockDim.x a multiple of 32, <= 1024).
// `warp_tot` is a 33-int shared scratch; returns this thread's exclusive
// prefix and writes the block total to *total.
__device__ __forceinline__ int block_excl_scan(int v, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int inc = warp_incl_scan(v, lane);
  if (lane == 31) warp_tot[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? warp_tot[lane] : 0;
    int wi = warp_incl_scan(w, lane);
    if (lane < nw) warp_tot[lane] = wi - w;
    if (lane == nw - 1) warp_tot[32] = wi;
  }
  __syncthreads();
  int res = warp_tot[warp] + inc - v;
  *total = warp_tot[32];
  __syncthreads();
  return res;
}

// Sum over the block; `warp_tot` is the same 33-int scratch as block_excl_scan.
__device__ __forceinline__ int block_sum(int v, int* warp_tot) {
  int total;
  block_excl_scan(v, warp_tot, &total);
  return total;
}

// ---------------------------------------------------------------------------
// Eq. 2 codes: round-half-even of the IEEE fp32 quotient v / gamma, clamped to
// +-qmax; gamma = 0 gives 0.
//
// quant_code divides exactly (__fdiv_rn).  quant_code_fast reaches the same
// integer from one correctly rounded reciprocal per row: t = v * fl(1/gamma)
// differs from v/gamma by at most ~2 ulp (|t - v/gamma| < 3.1e-5 for
// |v/gamma| <= 127.5), and the correctly rounded quotient Q lies within half
// an ulp (< 3.9e-6) of v/gamma, so |t - Q| < 3.5e-5.  rint(t) = rint(Q) unless
// a rounding boundary k + 1/2 lies within 4e-5 of t; only then (and for
// scales so small that 1/gamma is not finite) the exact division is taken.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int8_t quant_code(float v, float gamma, float qmax) {
  if (!(gamma > 0.f)) return 0;
  float q = rintf(__fdiv_rn(v, gamma));
  q = fminf(fmaxf(q, -qmax), qmax);
  return static_cast<int8_t>(static_cast<int>(q));
}

// inv = __fdiv_rn(1, gamma) for the row, computed once by the caller.  The
// rounding uses the fp32 adder: t + 1.5*2^23 rounds t to an integer (ties to
// even) for |t| < 2^22, and the sum's low bits are that integer.
__device__ __forceinline__ int quant_code_fast(float v, float gamma, float inv, float qmax) {
  if (!(gamma > 0.f)) return 0;
  const float t = v * inv;
  const float tb = t + 12582912.0f;  // 1.5 * 2^23
  const float r = tb - 12582912.0f;  // rint(t)
  int q;
  if (fabsf(fabsf(t - r) - 0.5f) < 4e-5f || !(fabsf(inv) < 3.0e38f)) {
    q = static_cast<int>(rintf(__fdiv_rn(v, gamma)));
  } else {
    q = __float_as_int(tb) - 0x4B400000;
  }
  const int qm = static_cast<int>(qmax);
  return q < -qm ? -qm : (q > qm ? qm : q);
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float (&f)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

__device__ __forceinline__ uint2 quant8(const float (&f)[8], float gamma, float qmax) {
  const float inv = gamma > 0.f ? __fdiv_rn(1.0f, gamma) : 0.f;
  uint32_t lo = 0, hi = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    lo |= static_cast<uint32_t>(static_cast<uint8_t>(quant_code_fast(f[i], gamma, inv, qmax))) << (8 * i);
    hi |= static_cast<uint32_t>(static_cast<uint8_t>(quant_code_fast(f[4 + i], gamma, inv, qmax))) << (8 * i);
  }
  return make_uint2(lo, hi);
}

// Eight codes of one 16-byte bf16 vector (the same rule as quant_code), in
// packed arithmetic: t = v * fl(1/gamma) rounded by the 1.5*2^23 adder, the
// code read from the low byte of the sum.  The whole vector takes the exact
// per-value path when gamma is not a positive finite scale, 1/gamma
// overflows, any |t| reaches qmax + 1/2 (a clamp), or any t lies within 4e-5 of a
// rounding boundary k + 1/2 (the bound of quant_code_fast).
__device__ __forceinline__ uint2 quant8_packed(const uint4& u, float gamma, float qmax) {
  float f[8];
  bf16x8_to_f32(u, f);
  const float inv = gamma > 0.f ? __fdiv_rn(1.0f, gamma) : 0.f;
  const float2 iv = make_float2(inv, inv);
  const float2 big = make_float2(12582912.0f, 12582912.0f), nbig = make_float2(-12582912.0f, -12582912.0f);
  uint32_t code[8];
  float dmax = 0.f, tmax = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = fmul2(make_float2(f[2 * i], f[2 * i + 1]), iv);
    const float2 tb = fadd2(t, big);
    const float2 r = fadd2(tb, nbig);
    dmax = fmax3(dmax, fabsf(t.x - r.x), fabsf(t.y - r.y));
    tmax = fmax3(tmax, fabsf(t.x), fabsf(t.y));
    code[2 * i] = __float_as_uint(tb.x);
    code[2 * i + 1] = __float_as_uint(tb.y);
  }
  if (gamma > 0.f && gamma < 3.0e38f && inv < 3.0e38f && dmax < 0.5f - 4e-5f && tmax < qmax + 0.5f) {
    const uint32_t lo = __byte_perm(__byte_perm(code[0], code[1], 0x0040), __byte_perm(code[2], code[3], 0x0040), 0x5410);
    const uint32_t hi = __byte_perm(__byte_perm(code[4], code[5], 0x0040), __byte_perm(code[6], code[7], 0x0040), 0x5410);
    return make_uint2(lo, hi);
  }
  uint32_t lo = 0, hi = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    lo |= static_cast<uint32_t>(static_cast<uint8_t>(quant_code(f[i], gamma, qmax))) << (8 * i);
    hi |= static_cast<uint32_t>(static_cast<uint8_t>(quant_code(f[4 + i], gamma, qmax))) << (8 * i);
  }
  return make_uint2(lo, hi);
}

// The eight codes of quant8_packed (qmax <= 7) stored as 4-bit two's
// complement, two per byte: code 2i in the low nibble of byte i, code 2i+1 in
// its high nibble.
__device__ __forceinline__ uint32_t quant4_packed(const uint4& u, float gamma, float qmax) {
  const uint2 c = quant8_packed(u, gamma, qmax);
  // bytes b0..b3 of a word -> nibbles: (b0 | b1 << 4) in byte 0, (b2 | b3 << 4) in byte 2
  const uint32_t x = c.x & 0x0F0F0F0Fu, y = c.y & 0x0F0F0F0Fu;
  const uint32_t xs = x | (x >> 4), ys = y | (y >> 4);
  return __byte_perm(xs, ys, 0x6420);
}

__device__ __forceinline__ uint2 quant8_bf16(const uint4& u, float gamma, float qmax) {
  float f[8];
  bf16x8_to_f32(u, f);
  return quant8(f, gamma, qmax);
}

}  // namespace tp
