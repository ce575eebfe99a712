// ptx.cuh -- thin inline-PTX wrappers for sm_103a: mbarriers (with bounded waits), TMA,
// tcgen05 (TMEM allocation, MMA, commit, loads), fences and cluster shared memory.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace qwam {

// Sticky device error bits (written to the handle's error word).
enum : int { kErrTimeout = 1, kErrRange = 2 };

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t warp_id() { return threadIdx.x >> 5; }
__device__ __forceinline__ uint32_t lane_id() { return threadIdx.x & 31; }

__device__ __forceinline__ bool elect_one() {
  uint32_t pred = 0;
  asm volatile(
      "{\n.reg .b32 rx;\n.reg .pred px;\n"
      "elect.sync rx|px, 0xffffffff;\n"
      "selp.u32 %0, 1, 0, px;\n}"
      : "=r"(pred));
  return pred != 0;
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("{\n.reg .b64 st;\nmbarrier.arrive.shared::cta.b64 st, [%0];\n}" ::"r"(smem_u32(bar)) : "memory");
}
// One arrival for the whole warp once all of its lanes are here (each lane has issued its own
// fences before calling).  Barriers that warps release are initialised with a count of warps:
// per-thread arrivals on a shared barrier serialise and cost more than the work they guard.
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("{\n.reg .b64 st;\nmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking test of a phase (never suspends): issued early, its result is consumed later, so
// that its latency overlaps independent work.
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\n"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Every wait in the kernels is bounded.  A kernel gives up when its deadline passes or when
// another warp of the CTA has already given up (shared abort flag); it then records
// kErrTimeout in the error word and unwinds.
struct WaitCtl {
  volatile int* abort_flag;  // shared memory, 0 = running
  int* err;                  // global error word (first error kept until read)
  uint64_t deadline_ns;      // %globaltimer value after which waits give up
};

// try_wait with a suspend-time hint: a thread whose phase is not complete sleeps until it
// completes or `ns` nanoseconds pass, instead of polling and taking issue slots from the warps
// that do the work.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t ns) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      "selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(ns)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool wait_loop(uint64_t* bar, uint32_t parity, const WaitCtl& c) {
  for (;;) {
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if (*c.abort_flag) return false;
    if (globaltimer_ns() > c.deadline_ns) {
      *c.abort_flag = 1;
      atomicOr(c.err, kErrTimeout);
      return false;
    }
  }
}
static __device__ __noinline__ bool wait_slow(uint64_t* bar, uint32_t parity, const WaitCtl& c) {
  return wait_loop(bar, parity, c);
}
// Every lane that calls a wait together gets the same answer: a lane that saw the phase complete
// and one that gave up at the deadline would otherwise part ways before a warp-wide instruction
// (elect.sync, a warp barrier) that needs them all.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, const WaitCtl& c) {
  const bool r = mbar_try_wait(bar, parity) || wait_slow(bar, parity, c);
  return __all_sync(__activemask(), r) != 0;
}
// The same wait with the slow loop inlined, for kernels that set per-warpgroup register budgets
// (setmaxnreg): ptxas cannot allocate registers for a function called from such regions.  It is
// on the hot paths, so it takes no vote: a warp that enters it converged stays converged, because
// each try is one warp instruction on one barrier (every lane gets the same result) and the loop's
// deadline checks fall on the same iteration for every lane.
__device__ __forceinline__ bool mbar_wait_inline(uint64_t* bar, uint32_t parity, const WaitCtl& c) {
  if (mbar_try_wait(bar, parity)) return true;
  return wait_loop(bar, parity, c);
}

// ---------------------------------------------------------------- programmatic dependent launch
// The layer's kernels are launched with programmatic stream serialization: each lets the next
// kernel of the stream be scheduled as soon as it starts (its CTAs then set up barriers and
// tensor memory while this one runs), and waits, before it touches global memory, until the
// previous kernel has completed and its writes are visible.
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// ---------------------------------------------------------------- fences
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void named_bar_sync(uint32_t id, uint32_t nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// ---------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* m) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}
// 2D tiled load; x = innermost coordinate (elements), y = row.  x * elemsize must be a
// multiple of 16 bytes (all callers pass multiples of the 16-byte box width).
__device__ __forceinline__ void tma_load_2d(void* smem_dst, const CUtensorMap* m, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

// 3D tiled load; x = innermost coordinate (elements, same 16-byte rule as above), then y, z.
__device__ __forceinline__ void tma_load_3d(void* smem_dst, const CUtensorMap* m, uint64_t* bar, int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z)
      : "memory");
}

// Non-tensor bulk copy global -> shared, completing `bytes` of transaction on `bar`.  Both
// addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load_1d(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(smem_dst)),
               "l"(reinterpret_cast<uint64_t>(gsrc)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// 2D tiled store shared -> global (bulk async-group completion).  x, y >= 0 (a store never
// starts at a negative coordinate), x * elemsize a multiple of 16 bytes; the part of the box
// outside the tensor's extent is not written.  The shared source must not change until
// bulk_wait_read() has returned in the issuing thread.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* m, const void* smem_src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(m)),
               "r"(smem_u32(smem_src)), "r"(x), "r"(y)
               : "memory");
}
// The same for a 3D box (x, y, z >= 0).
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* m, const void* smem_src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(m)),
               "r"(smem_u32(smem_src)), "r"(x), "r"(y), "r"(z)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Orders the async proxy's completed global writes before the thread's later generic operations
// (a release that other threads acquire then covers them).
__device__ __forceinline__ void fence_proxy_async_all() { asm volatile("fence.proxy.async;" ::: "memory"); }
// The issuing thread's committed bulk stores have read their shared sources.
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// The issuing thread's committed bulk stores are complete (their writes performed).
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ---------------------------------------------------------------- cluster
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_smem(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ float4 ld_dsmem_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// ---------------------------------------------------------------- tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t* smem_result, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(smem_result)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Shared-memory matrix descriptor (tcgen05): start, leading/stride byte offsets, layout.
enum : uint32_t { kSwNone = 0, kSw128 = 2, kSw64 = 4, kSw32 = 6 };
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo, uint32_t layout) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;  // descriptor version
  d |= static_cast<uint64_t>(layout) << 61;
  return d;
}

// Instruction descriptors: D = f32, A and B K-major.
__host__ __device__ constexpr uint32_t idesc_e4m3(int M, int N) {
  return (1u << 4) | (0u << 7) | (0u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}
__host__ __device__ constexpr uint32_t idesc_f16(int M, int N) {
  return (1u << 4) | (0u << 7) | (0u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

// Block-scaled FP4: A and B E2M1 (format code 1), scale factors UE4M3 (scale-format bit 23 = 0),
// scale-factor data IDs 0, M >> 7 in bits 27..28 (M = 128 or 256).
__host__ __device__ constexpr uint32_t idesc_nvf4(int M, int N) {
  return (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 7) << 27);
}

__device__ __forceinline__ void mma_f8f6f4(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D (+)= sum over K = 64 of (a sa)(b sb): E2M1 operands from shared memory, one UE4M3 scale per
// 16 K for every row of A (TMEM at sfa) and column of B (TMEM at sfb).  Row m of A takes its four
// scales from lane m, column sfa + m / 32; column n of B from lane 32 (m / 32) + n % 32, column
// sfb + n / 32 -- the placement tcgen05.cp.32x128b.warpx4 produces from a 512-byte atom.
__device__ __forceinline__ void mma_nvf4(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t sfa,
                                         uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %6, 0;\n"
      "tcgen05.mma.cta_group::1.kind::mxf4nvf4.block_scale.scale_vec::4X [%0], %1, %2, %3, [%4], [%5], p;\n}" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}
// Copy 32 rows x 16 bytes of shared memory (no swizzle, rows contiguous) into TMEM lanes
// 0..31 of every lane quarter, four 32-bit columns from `taddr`.
__device__ __forceinline__ void tc_cp_32x128b_x4(uint32_t taddr, uint64_t sdesc) {
  asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(sdesc) : "memory");
}
// Arrive once on `bar` when all previously issued tcgen05.mma of this thread have completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// 32 TMEM lanes x 32 consecutive 32-bit columns: thread t gets lane (base + t), 32 values.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}
// 32 lanes x 16 columns.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// The same wait, naming the 32 registers of one tcgen05.ld as its operands: the compiler then
// cannot move a use of those registers above the wait, so loads can be issued ahead (software
// pipelining) while other registers are being consumed.
__device__ __forceinline__ void tmem_ld_wait_dep(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}

// tcgen05.ld.16x256b.x4: 16 TMEM lanes x 32 columns.  Thread t receives register 4j + q =
// (lane t/4 + 8 [q >= 2], column 8j + 2 (t % 4) + (q & 1)), j = 0..3: four threads share a lane
// (row) and eight share a column pair.
__device__ __forceinline__ void tmem_ld16x256_x4(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x4.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
// Wait for outstanding tcgen05.ld, naming both destination arrays (see tmem_ld_wait_dep).
__device__ __forceinline__ void tmem_ld_wait_dep2(uint32_t (&a)[16], uint32_t (&b)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(a[0]), "+r"(a[1]), "+r"(a[2]), "+r"(a[3]), "+r"(a[4]), "+r"(a[5]), "+r"(a[6]), "+r"(a[7]),
                 "+r"(a[8]), "+r"(a[9]), "+r"(a[10]), "+r"(a[11]), "+r"(a[12]), "+r"(a[13]), "+r"(a[14]),
                 "+r"(a[15]), "+r"(b[0]), "+r"(b[1]), "+r"(b[2]), "+r"(b[3]), "+r"(b[4]), "+r"(b[5]), "+r"(b[6]),
                 "+r"(b[7]), "+r"(b[8]), "+r"(b[9]), "+r"(b[10]), "+r"(b[11]), "+r"(b[12]), "+r"(b[13]),
                 "+r"(b[14]), "+r"(b[15])
               :
               : "memory");
}

// Wait for outstanding tcgen05.ld and hand the two 16-register results on as 16 packed pairs
// p[i] = {r[2i], r[2i + 1]} (a then b): the pairing happens after the wait, in the form the
// register allocator maps onto aligned register pairs.
__device__ __forceinline__ void tmem_ld_wait_pairs(const uint32_t (&a)[16], const uint32_t (&b)[16],
                                                   unsigned long long (&p)[16]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;\n"
      "mov.b64 %0, {%16, %17};\n"
      "mov.b64 %1, {%18, %19};\n"
      "mov.b64 %2, {%20, %21};\n"
      "mov.b64 %3, {%22, %23};\n"
      "mov.b64 %4, {%24, %25};\n"
      "mov.b64 %5, {%26, %27};\n"
      "mov.b64 %6, {%28, %29};\n"
      "mov.b64 %7, {%30, %31};\n"
      "mov.b64 %8, {%32, %33};\n"
      "mov.b64 %9, {%34, %35};\n"
      "mov.b64 %10, {%36, %37};\n"
      "mov.b64 %11, {%38, %39};\n"
      "mov.b64 %12, {%40, %41};\n"
      "mov.b64 %13, {%42, %43};\n"
      "mov.b64 %14, {%44, %45};\n"
      "mov.b64 %15, {%46, %47};\n"
      : "=l"(p[0]), "=l"(p[1]), "=l"(p[2]), "=l"(p[3]), "=l"(p[4]), "=l"(p[5]), "=l"(p[6]), "=l"(p[7]), "=l"(p[8]), "=l"(p[9]), "=l"(p[10]), "=l"(p[11]), "=l"(p[12]), "=l"(p[13]), "=l"(p[14]), "=l"(p[15])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(a[4]), "r"(a[5]), "r"(a[6]), "r"(a[7]), "r"(a[8]), "r"(a[9]), "r"(a[10]), "r"(a[11]), "r"(a[12]), "r"(a[13]), "r"(a[14]), "r"(a[15]), "r"(b[0]), "r"(b[1]), "r"(b[2]), "r"(b[3]), "r"(b[4]), "r"(b[5]), "r"(b[6]), "r"(b[7]), "r"(b[8]), "r"(b[9]), "r"(b[10]), "r"(b[11]), "r"(b[12]), "r"(b[13]), "r"(b[14]), "r"(b[15])
      : "memory");
}
// Wait for outstanding tcgen05.ld and hand one 16-register result on as 8 packed pairs
// p[i] = {r[2i], r[2i + 1]}.
__device__ __forceinline__ void tmem_ld_wait_pairs8(const uint32_t (&a)[16], unsigned long long (&p)[8]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;\n"
      "mov.b64 %0, {%8, %9};\n"
      "mov.b64 %1, {%10, %11};\n"
      "mov.b64 %2, {%12, %13};\n"
      "mov.b64 %3, {%14, %15};\n"
      "mov.b64 %4, {%16, %17};\n"
      "mov.b64 %5, {%18, %19};\n"
      "mov.b64 %6, {%20, %21};\n"
      "mov.b64 %7, {%22, %23};\n"
      : "=l"(p[0]), "=l"(p[1]), "=l"(p[2]), "=l"(p[3]), "=l"(p[4]), "=l"(p[5]), "=l"(p[6]), "=l"(p[7])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(a[4]), "r"(a[5]), "r"(a[6]), "r"(a[7]), "r"(a[8]),
        "r"(a[9]), "r"(a[10]), "r"(a[11]), "r"(a[12]), "r"(a[13]), "r"(a[14]), "r"(a[15])
      : "memory");
}
// Wait for outstanding tcgen05.ld and hand four 16-register results on as packed pairs
// p[i][j] = {r[i][2j], r[i][2j + 1]}.
__device__ __forceinline__ void tmem_ld_wait_pairs8x4(const uint32_t (&a)[4][16], unsigned long long (&p)[4][8]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;\n"
      "mov.b64 %0, {%32, %33};\n mov.b64 %1, {%34, %35};\n mov.b64 %2, {%36, %37};\n mov.b64 %3, {%38, %39};\n"
      "mov.b64 %4, {%40, %41};\n mov.b64 %5, {%42, %43};\n mov.b64 %6, {%44, %45};\n mov.b64 %7, {%46, %47};\n"
      "mov.b64 %8, {%48, %49};\n mov.b64 %9, {%50, %51};\n mov.b64 %10, {%52, %53};\n mov.b64 %11, {%54, %55};\n"
      "mov.b64 %12, {%56, %57};\n mov.b64 %13, {%58, %59};\n mov.b64 %14, {%60, %61};\n mov.b64 %15, {%62, %63};\n"
      "mov.b64 %16, {%64, %65};\n mov.b64 %17, {%66, %67};\n mov.b64 %18, {%68, %69};\n mov.b64 %19, {%70, %71};\n"
      "mov.b64 %20, {%72, %73};\n mov.b64 %21, {%74, %75};\n mov.b64 %22, {%76, %77};\n mov.b64 %23, {%78, %79};\n"
      "mov.b64 %24, {%80, %81};\n mov.b64 %25, {%82, %83};\n mov.b64 %26, {%84, %85};\n mov.b64 %27, {%86, %87};\n"
      "mov.b64 %28, {%88, %89};\n mov.b64 %29, {%90, %91};\n mov.b64 %30, {%92, %93};\n mov.b64 %31, {%94, %95};\n"
      : "=l"(p[0][0]), "=l"(p[0][1]), "=l"(p[0][2]), "=l"(p[0][3]), "=l"(p[0][4]), "=l"(p[0][5]), "=l"(p[0][6]),
        "=l"(p[0][7]), "=l"(p[1][0]), "=l"(p[1][1]), "=l"(p[1][2]), "=l"(p[1][3]), "=l"(p[1][4]), "=l"(p[1][5]),
        "=l"(p[1][6]), "=l"(p[1][7]), "=l"(p[2][0]), "=l"(p[2][1]), "=l"(p[2][2]), "=l"(p[2][3]), "=l"(p[2][4]),
        "=l"(p[2][5]), "=l"(p[2][6]), "=l"(p[2][7]), "=l"(p[3][0]), "=l"(p[3][1]), "=l"(p[3][2]), "=l"(p[3][3]),
        "=l"(p[3][4]), "=l"(p[3][5]), "=l"(p[3][6]), "=l"(p[3][7])
      : "r"(a[0][0]), "r"(a[0][1]), "r"(a[0][2]), "r"(a[0][3]), "r"(a[0][4]), "r"(a[0][5]), "r"(a[0][6]),
        "r"(a[0][7]), "r"(a[0][8]), "r"(a[0][9]), "r"(a[0][10]), "r"(a[0][11]), "r"(a[0][12]), "r"(a[0][13]),
        "r"(a[0][14]), "r"(a[0][15]), "r"(a[1][0]), "r"(a[1][1]), "r"(a[1][2]), "r"(a[1][3]), "r"(a[1][4]),
        "r"(a[1][5]), "r"(a[1][6]), "r"(a[1][7]), "r"(a[1][8]), "r"(a[1][9]), "r"(a[1][10]), "r"(a[1][11]),
        "r"(a[1][12]), "r"(a[1][13]), "r"(a[1][14]), "r"(a[1][15]), "r"(a[2][0]), "r"(a[2][1]), "r"(a[2][2]),
        "r"(a[2][3]), "r"(a[2][4]), "r"(a[2][5]), "r"(a[2][6]), "r"(a[2][7]), "r"(a[2][8]), "r"(a[2][9]),
        "r"(a[2][10]), "r"(a[2][11]), "r"(a[2][12]), "r"(a[2][13]), "r"(a[2][14]), "r"(a[2][15]), "r"(a[3][0]),
        "r"(a[3][1]), "r"(a[3][2]), "r"(a[3][3]), "r"(a[3][4]), "r"(a[3][5]), "r"(a[3][6]), "r"(a[3][7]),
        "r"(a[3][8]), "r"(a[3][9]), "r"(a[3][10]), "r"(a[3][11]), "r"(a[3][12]), "r"(a[3][13]), "r"(a[3][14]),
        "r"(a[3][15])
      : "memory");
}
// Wait for outstanding tcgen05.ld, naming four 16-register results as its operands (see
// tmem_ld_wait_dep: no use of those registers moves above the wait).
__device__ __forceinline__ void tmem_ld_wait_dep4(uint32_t (&a)[4][16]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+r"(a[0][0]), "+r"(a[0][1]), "+r"(a[0][2]), "+r"(a[0][3]), "+r"(a[0][4]), "+r"(a[0][5]), "+r"(a[0][6]),
        "+r"(a[0][7]), "+r"(a[0][8]), "+r"(a[0][9]), "+r"(a[0][10]), "+r"(a[0][11]), "+r"(a[0][12]), "+r"(a[0][13]),
        "+r"(a[0][14]), "+r"(a[0][15]), "+r"(a[1][0]), "+r"(a[1][1]), "+r"(a[1][2]), "+r"(a[1][3]), "+r"(a[1][4]),
        "+r"(a[1][5]), "+r"(a[1][6]), "+r"(a[1][7]), "+r"(a[1][8]), "+r"(a[1][9]), "+r"(a[1][10]), "+r"(a[1][11]),
        "+r"(a[1][12]), "+r"(a[1][13]), "+r"(a[1][14]), "+r"(a[1][15]), "+r"(a[2][0]), "+r"(a[2][1]), "+r"(a[2][2]),
        "+r"(a[2][3]), "+r"(a[2][4]), "+r"(a[2][5]), "+r"(a[2][6]), "+r"(a[2][7]), "+r"(a[2][8]), "+r"(a[2][9]),
        "+r"(a[2][10]), "+r"(a[2][11]), "+r"(a[2][12]), "+r"(a[2][13]), "+r"(a[2][14]), "+r"(a[2][15]), "+r"(a[3][0]),
        "+r"(a[3][1]), "+r"(a[3][2]), "+r"(a[3][3]), "+r"(a[3][4]), "+r"(a[3][5]), "+r"(a[3][6]), "+r"(a[3][7]),
        "+r"(a[3][8]), "+r"(a[3][9]), "+r"(a[3][10]), "+r"(a[3][11]), "+r"(a[3][12]), "+r"(a[3][13]), "+r"(a[3][14]),
        "+r"(a[3][15])
      :
      : "memory");
}
// {x, x} as a packed pair.
__device__ __forceinline__ unsigned long long dup2(float x) {
  unsigned long long d;
  asm("mov.b64 %0, {%1, %1};" : "=l"(d) : "f"(x));
  return d;
}

// Per-warpgroup register budgets (all four warps of a warpgroup execute the same instruction).
// The sum over the CTA's warps must not exceed what the CTA was launched with (threads x the
// kernel's register count), or an increase would wait for registers that never come free.
template <uint32_t N>
__device__ __forceinline__ void setmaxnreg_dec() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}
template <uint32_t N>
__device__ __forceinline__ void setmaxnreg_inc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

}  // namespace qwam
