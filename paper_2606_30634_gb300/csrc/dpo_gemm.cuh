// dpo_gemm.cuh -- batched bf16 GEMM on the sm_103a tensor cores (tcgen05,
// TMA, TMEM) with the epilogues of the Newton-Schulz iteration.
//
//   D[b] = alpha * A[b] B[b]^T + beta * C[b]      (optionally also D[b]^T)
//
// A[b] (M x K) and B[b] (N x K) are row-major bf16 ("K-major" operands), the
// product accumulates in fp32 in tensor memory, and the epilogue rounds once
// to bf16. Every dimension is a multiple of the tile (the Newton-Schulz
// scratch is padded with zeros to multiples of 256), so no tile is partial.
//
// A persistent grid of CTA pairs (clusters of 2, one CTA per SM) walks the
// 256 x 256 output tiles with the 2-SM MMA. In each CTA:
//   warp 0      TMA producer: this CTA's 128 x 128 half of the A block and
//               128 x 128 half of the B block (bf16, 128-byte swizzle, two
//               64-wide boxes each) into a 3-stage ring, completing on the
//               leader CTA's mbarrier;
//   warp 1      allocates 512 TMEM columns (two accumulators) together with
//               the peer; in the leader, one lane issues
//               tcgen05.mma.cta_group::2.kind::f16 (M 256, N 256, K 16) eight
//               times per stage, reading both CTAs' halves, and commits each
//               stage and each finished tile to both CTAs;
//   warps 2-5   epilogue of this CTA's 128 rows: tcgen05.ld 32 lanes x 32
//               columns at a time, scale, add the addend, round to bf16,
//               stage the 32 x 32 chunk (and, when asked, its transpose) in
//               shared memory and write it with a TMA store.
// Per CTA a stage is 64 KiB for 8.4 MFLOP, a third less than one SM holding
// a whole 128 x 256 operand pair, so three stages fit and keep the tensor
// pipe fed across the L2 / DRAM round trip.
// Symmetric products (Params::sym; X X^T and c A A + b A): only tiles on or
// above the diagonal block (n0 >= m0) are computed; each of their
// elements (i, j) is also stored at (j, i) when the tile holding (j, i) is
// not computed. Every element is then written exactly once, by one thread,
// and the result does not depend on scheduling.
// Every wait on an mbarrier gives up after kWaitNs, records an error code and
// lets the CTA finish (draining its own TMA loads first), so a fault in the
// pipeline surfaces as a status instead of a hang.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cstdint>

namespace dpo {
namespace gemm {

// A CTA pair (a cluster of 2) computes one TM x TN output tile with the
// 2-SM MMA: each CTA holds BM = TM / 2 rows of A and BH = TN / 2 rows of B
// per stage, and its TMEM holds its BM rows of the accumulator. A stage
// spans BK = 128 of K as two TMA boxes of kBoxK = 64 (the 128-byte swizzle
// span); eight MMAs per stage halve the barrier hand-offs per MMA against
// 64-wide stages, which measured 10% faster on GB300 at equal ring size.
constexpr int TM = 256, TN = 256, BM = 128, BH = 128, BK = 128, kBoxK = 64, kStages = 3;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 256;                  // one accumulator (fp32, TN columns)
constexpr int kABytes = BM * BK * 2;                 // 32 KiB
constexpr int kBBytes = BH * BK * 2;                 // 32 KiB
constexpr int kStageBytes = kABytes + kBBytes;       // 64 KiB per CTA
// Epilogue staging behind the ring: per epilogue warp two buffers for its
// 32 x 32 chunk of D and two for the chunk's transpose, 2 KiB each, in the
// 64-byte-swizzled layout the TMA store reads.
constexpr int kChunkBytes = 32 * 32 * 2;
constexpr int kEpiBytes = 4 * 4 * kChunkBytes;              // 32 KiB
// ring + 1024-byte alignment slack + staging
constexpr int kSmemBytes = kStages * kStageBytes + 1024 + kEpiBytes;
constexpr unsigned long long kWaitNs = 1000000000ull;  // 1 s per wait

// Error codes OR-ed into Params::err (kErrWaitDone: an accumulator hand-off).
constexpr unsigned int kErrWaitFull = 1u, kErrWaitEmpty = 2u, kErrWaitDone = 4u,
                       kErrDrain = 8u;

// D is written through the group's store map d (boxes of 32 x 32, 64-byte
// swizzle) and, with trans, D^T through dt.
struct Params {
    const __nv_bfloat16 *c;       // M x N addend, or nullptr
    int64_t ldc, c_bstride;
    float alpha, beta;
    int k_blocks;                 // K / BK
    int sym;                      // D is symmetric (M == N): see ns_gemm_kernel
    int trans;                    // also write D^T (N x M) through the map dt
    int stall;                    // test hook: the MMA lane's first accumulator wait
                                  // targets a phase no arrival completes, so it gives up
    unsigned int *err;
};

__device__ __forceinline__ unsigned long long globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the phase with the given parity to complete, for at most kWaitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    if (mbar_try(bar, parity))
        return true;
    const unsigned long long t0 = globaltimer();
    while (!mbar_try(bar, parity))
        if (globaltimer() - t0 > kWaitNs)
            return false;
    return true;
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

// TMA tile load into this CTA's shared memory; the mbarrier (a shared::cluster
// address) may belong to either CTA of the pair.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int x, int y,
                                            int z, uint32_t bar_cluster)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar_cluster)
        : "memory");
}

// TMA store of a 32 x 32 bf16 box from this CTA's shared memory to global
// coordinates (x = column, y = row, z = batch entry), in this thread's bulk
// async-group.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap *map, uint32_t src, int x, int y,
                                             int z)
{
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];"
                 ::"l"(reinterpret_cast<uint64_t>(map)), "r"(src), "r"(x), "r"(y), "r"(z)
                 : "memory");
}

// Byte offset of 16-byte granule g of row r in a tile of 64-byte rows with
// the 64-byte swizzle (granule index XOR bits 1-2 of the row).
__device__ __forceinline__ uint32_t swz64(int r, int g)
{
    return (uint32_t)(r * 64 + ((g ^ ((r >> 1) & 3)) << 4));
}

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// shared::cluster address of the same shared::cta offset in CTA `rank`
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cluster)
{
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster)
                 : "memory");
}

__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored as rows of
// 64 bf16 (128 bytes) with the 128-byte swizzle, 8-row groups 1024 bytes
// apart (the layout the TMA box above produces): start address, leading
// byte offset 16 (unused by swizzled K-major layouts), stride byte offset
// 1024, descriptor version 1, swizzle mode 2 (128-byte).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr)
{
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)(16 >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// Shared-memory descriptor of an MN-major operand tile: rows of 64 bf16
// (128 bytes) along N with the 128-byte swizzle, one row per K index, 8-row
// K groups 1024 bytes apart (stride byte offset), and the second 64-column
// N chunk 8192 bytes further (leading byte offset: one 64-row TMA box).
__device__ __forceinline__ uint64_t smem_desc_mn(uint32_t addr)
{
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)(8192 >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, A
// K-major, N = TN, M = TM (the pair's 2-SM shape); B K-major, or MN-major
// with bit 16 (B read as stored row-major along N).
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(TN >> 3) << 17) |
                            ((uint32_t)(TM >> 4) << 24);
constexpr uint32_t kIdescBmn = kIdesc | (1u << 16);

// One TM x TN x 16 step of the pair, issued by the leader CTA: A rows from
// both CTAs' shared memory at the descriptor's offset, B likewise, the
// accumulator rows in each CTA's TMEM.
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate));
}

// Arrive on the mbarrier at this shared::cta offset in both CTAs of the pair
// once the leader's MMAs issued so far have completed.
__device__ __forceinline__ void mma_commit_pair(uint32_t bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
        " [%0], %1;" ::"r"(bar), "h"((uint16_t)0x3)
        : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// Tile t of a launch: batch entry, row block and column block. A full
// product walks bands of kBandRows block rows (all of them, up to 4096 rows),
// each band column by column, so the tiles in flight at once (one per CTA
// pair) share the band's A row blocks and a few B column blocks in L2, and
// each B column block comes from DRAM about once per band. On a 4096 x 11008
// operand, walking whole block rows instead had the pairs stream all 43 B
// column blocks every round. A symmetric product (sym, m_tiles == n_tiles)
// enumerates only the tiles on or above the diagonal, column by column
// (column n holds n + 1 of them), so the pairs' shares of its work differ by
// at most one tile, and the tiles in flight at once read the first block rows
// of the operand before the pairs move on to the last ones.
constexpr int kBandRows = 16;   // block rows per band of a full product's walk

struct TileGrid {
    int m_tiles, n_tiles, nb, sym;
    __host__ __device__ __forceinline__ int per_batch() const
    {
        return sym ? m_tiles * (m_tiles + 1) / 2 : m_tiles * n_tiles;
    }
    __host__ __device__ __forceinline__ int count() const { return per_batch() * nb; }
    __device__ __forceinline__ void at(int t, int &b, int &m0, int &n0) const
    {
        const int per = per_batch();
        b = t / per;
        int u = t - b * per;
        if (sym) {
            int n = 0;
            while (u > n) {   // u < per, so n stays below m_tiles
                u -= n + 1;
                ++n;
            }
            m0 = u * TM;
            n0 = n * TN;
        } else {
            const int band = u / (kBandRows * n_tiles);
            const int first = band * kBandRows;
            const int rows = min(kBandRows, m_tiles - first);
            const int r = u - first * n_tiles;   // 0 <= r < rows * n_tiles
            m0 = (first + r % rows) * TM;
            n0 = (r / rows) * TN;
        }
    }
};

// One launch computes the same product for up to kMaxGroups batches of
// different shapes (the shape groups of a Newton-Schulz step): each group
// has its own operand and output maps, epilogue and tile grid, and its tiles
// follow the previous group's in the launch's order. Small sets then fill
// the CTA pairs with one launch per product instead of one per shape.
constexpr int kMaxGroups = 4;

struct GemmGroup {
    CUtensorMap a, b, d, dt;   // A, B (operands), D and D^T (stores)
    Params p;
    TileGrid tg;
    int tile0;                 // first tile of this group in the launch
};

struct GemmLaunch {
    GemmGroup g[kMaxGroups];
    int n_groups;
    int n_tiles;               // over all groups
};

// Group, batch entry, row block and column block of tile t of a launch.
__device__ __forceinline__ const GemmGroup &locate(const GemmLaunch &L, int t, int &b, int &m0,
                                                   int &n0)
{
    int gi = L.n_groups - 1;
    while (gi > 0 && t < L.g[gi].tile0)
        --gi;
    const GemmGroup &G = L.g[gi];
    G.tg.at(t - G.tile0, b, m0, n0);
    return G;
}

// Persistent: the CTA pairs (clusters of 2) take tiles c, c + pairs, ...
// Within a pair, rank 0 (the leader) issues the MMAs; both ranks load their
// halves of A and B and drain their own accumulator rows. Two accumulators
// in TMEM (columns 0-255 and 256-511) let the MMA fill one while the
// epilogues drain the other.
//   full[s]      (leader) both ranks' TMA bytes of stage s have landed
//   empty[s]     (each)   the leader's MMAs have finished reading stage s
//   acc_full[a]  (each)   accumulator a holds a finished tile
//   acc_empty[a] (leader) all 8 epilogue warps of the pair have read it
// BMN: the B operand is stored N-contiguous (a row-major K x N matrix) and
// loaded as two 64 x 64 boxes per stage, read MN-major by the MMA.
template <bool BMN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    ns_gemm_kernel(const __grid_constant__ GemmLaunch L)
{
    const Params &p0 = L.g[0].p;   // err and stall are the launch's
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t bars[2 * kStages + 4];
    __shared__ uint32_t tmem_slot;
    __shared__ int aborted;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
    const uint32_t raw = (uint32_t)__cvta_generic_to_shared(smem_raw);
    const uint32_t ring = (raw + 1023u) & ~1023u;   // the swizzle atoms repeat every 1024 B
    const uint32_t sa = ring, sb = ring + kStages * kABytes;
    const uint32_t bar0 = (uint32_t)__cvta_generic_to_shared(bars);
    auto full = [&](int s) { return bar0 + 8u * (uint32_t)s; };
    auto empty = [&](int s) { return bar0 + 8u * (uint32_t)(kStages + s); };
    auto acc_full = [&](int a) { return bar0 + 8u * (uint32_t)(2 * kStages + a); };
    auto acc_empty = [&](int a) { return bar0 + 8u * (uint32_t)(2 * kStages + 2 + a); };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(full(s), 1);
            mbar_init(empty(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(acc_full(a), 1);
            mbar_init(acc_empty(a), 8);   // one arrival per epilogue warp of the pair
        }
        aborted = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {   // both CTAs of the pair allocate together
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         (uint32_t)__cvta_generic_to_shared(&tmem_slot)),
                     "r"(2 * kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    cluster_sync();   // barriers of both CTAs initialised before any remote use
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_slot;
    const int n_tiles = L.n_tiles;

    if (warp == 0) {
        if (lane == 0) {
            for (int gi = 0; gi < L.n_groups; ++gi) {
                asm volatile("prefetch.tensormap [%0];"
                             ::"l"(reinterpret_cast<uint64_t>(&L.g[gi].a)) : "memory");
                asm volatile("prefetch.tensormap [%0];"
                             ::"l"(reinterpret_cast<uint64_t>(&L.g[gi].b)) : "memory");
            }
            int it = 0;   // k-blocks issued by this CTA
            for (int t = pair; t < n_tiles && !*(volatile int *)&aborted; t += n_pairs) {
                int b, m0, n0;
                const GemmGroup &G = locate(L, t, b, m0, n0);
                const CUtensorMap *tma_a = &G.a, *tma_b = &G.b;
                const int kb_n = G.p.k_blocks;
                const int ma = m0 + (int)rank * BM, nb_ = n0 + (int)rank * BH;
                for (int kb = 0; kb < kb_n; ++kb, ++it) {
                    const int s = it % kStages;
                    const uint32_t ph = (uint32_t)(it / kStages) & 1u;
                    if (!mbar_wait(empty(s), ph ^ 1u) || *(volatile int *)&aborted) {
                        atomicOr(p0.err, kErrWaitEmpty);
                        aborted = 1;
                        break;
                    }
                    const uint32_t fbar = map_to_rank(full(s), 0);
                    if (leader)   // the leader's barrier counts both CTAs' bytes
                        mbar_arrive_expect_tx(full(s), (uint32_t)(2 * kStageBytes));
#pragma unroll
                    for (int h = 0; h < BK / kBoxK; ++h) {   // the two 64-wide K halves
                        const int k0 = kb * BK + h * kBoxK;
                        const uint32_t ah = sa + (uint32_t)(s * kABytes + h * (kABytes / 2));
                        const uint32_t bh = sb + (uint32_t)(s * kBBytes + h * (kBBytes / 2));
                        tma_load_3d(ah, tma_a, k0, ma, b, fbar);
                        if (BMN) {   // two 64 x 64 boxes: N columns nb_.. and nb_ + 64..
                            tma_load_3d(bh, tma_b, nb_, k0, b, fbar);
                            tma_load_3d(bh + (uint32_t)(kBBytes / 4), tma_b, nb_ + 64, k0, b, fbar);
                        } else {
                            tma_load_3d(bh, tma_b, k0, nb_, b, fbar);
                        }
                    }
                }
            }
            // Drain (leader): every stage issued by either CTA has landed
            // before the pair leaves (the peer waits at the final cluster
            // barrier for this).
            if (leader)
                for (int q = it - kStages < 0 ? 0 : it - kStages; q < it; ++q)
                    if (!mbar_wait(full(q % kStages), (uint32_t)(q / kStages) & 1u))
                        atomicOr(p0.err, kErrDrain);
        }
    } else if (warp == 1) {
        if (lane == 0 && leader) {
            int it = 0, lt = 0;   // k-blocks consumed, tiles accumulated
            for (int t = pair; t < n_tiles && !*(volatile int *)&aborted; t += n_pairs) {
                int b, m0, n0;
                const int kb_n = locate(L, t, b, m0, n0).p.k_blocks;
                const int a = lt & 1;
                const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
                if (!mbar_wait(acc_empty(a), p0.stall && lt == 0 ? aph : aph ^ 1u)) {
                    atomicOr(p0.err, kErrWaitDone);
                    aborted = 1;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t d = tmem + (uint32_t)(a * (int)kTmemCols);
                bool ok = true;
                for (int kb = 0; kb < kb_n; ++kb, ++it) {
                    const int s = it % kStages;
                    const uint32_t ph = (uint32_t)(it / kStages) & 1u;
                    if (!mbar_wait(full(s), ph) || *(volatile int *)&aborted) {
                        atomicOr(p0.err, kErrWaitFull);
                        aborted = 1;
                        ok = false;
                        break;
                    }
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        const int h = k / (kBoxK / 16), kk = k % (kBoxK / 16);
                        const uint32_t ah = sa + (uint32_t)(s * kABytes + h * (kABytes / 2));
                        const uint32_t bh = sb + (uint32_t)(s * kBBytes + h * (kBBytes / 2));
                        const uint64_t ad = smem_desc(ah + (uint32_t)(kk * 32));
                        const uint64_t bd = BMN ? smem_desc_mn(bh + (uint32_t)(kk * 16 * 128))
                                                : smem_desc(bh + (uint32_t)(kk * 32));
                        mma_bf16(d, ad, bd, BMN ? kIdescBmn : kIdesc, (kb | k) != 0 ? 1u : 0u);
                    }
                    mma_commit_pair(empty(s));
                }
                mma_commit_pair(acc_full(a));   // when this tile's MMAs have completed
                ++lt;
                if (!ok) {
                    // the MMAs issued for this tile finish before the pair
                    // leaves and its TMEM is released
                    if (!mbar_wait(acc_full(a), aph))
                        atomicOr(p0.err, kErrDrain);
                    break;
                }
            }
        }
    } else {
        // Epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31 = this CTA's
        // tile rows m0 + BM rank + 32 (w % 4) + lane. Each 32 x 32 chunk is
        // staged in shared memory (and its transpose, for a mirrored or a
        // transposed output) and written by one TMA store per box from lane
        // 0; direct stores from 32 rows at a time cost the MMAs a fifth of
        // their rate on GB300. Two buffers per kind alternate, so lane 0
        // waits for the group of two chunks back before they are rewritten.
        const int q = warp & 3;
        const uint32_t wbuf = ring + (uint32_t)(kStages * kStageBytes + q * 4 * kChunkBytes);
        // The addend C (c A A + b A, B X + a X) is read kCPre chunks ahead of
        // its use, the first ones before the accumulator is ready, coalesced:
        // lane l loads granule l % 4 (8 columns) of rows l / 4 + 8 i of the
        // warp's 32 x 32 chunk, 8 rows of 64 bytes per instruction; the chunk
        // is then turned through its staging buffer so that each lane holds
        // its own row. Loading each lane's own row instead touched 32 lines
        // per instruction; where K is short (768) that made the chain 6 %
        // slower on GB300, and where K is long the epilogue is hidden behind
        // the MMAs either way. C is never the launch's output.
        constexpr int kCPre = 4;
        const int crs = lane >> 2, cg = lane & 3;   // coalesced load: sub-row, granule
        int lt = 0, staged = 0;
        for (int t = pair; t < n_tiles; t += n_pairs) {
            int b, m0, n0;
            const GemmGroup &G = locate(L, t, b, m0, n0);
            const Params &p = G.p;
            const int a = lt & 1;
            const int row0 = m0 + (int)rank * BM + q * 32;
            // C at (row0 + crs, n0 + 8 cg); rows 8 i further for i = 0..3
            const __nv_bfloat16 *crow =
                p.c != nullptr ? p.c + (int64_t)b * p.c_bstride + (int64_t)(row0 + crs) * p.ldc +
                                     n0 + cg * 8
                               : nullptr;
            const int64_t c8 = 8 * p.ldc;
            uint4 cpre[kCPre][4];
            if (crow != nullptr) {
#pragma unroll
                for (int c = 0; c < kCPre; ++c)
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        cpre[c][i] = __ldg(reinterpret_cast<const uint4 *>(crow + i * c8 + c * 32));
            }
            const bool seen = mbar_wait(acc_full(a), (uint32_t)(lt >> 1) & 1u);
            if (!seen)
                atomicOr(p0.err, kErrWaitDone);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            // tcgen05.ld is warp-collective: the whole warp goes on, or none of it.
            if (!__all_sync(0xFFFFFFFFu, seen && !*(volatile int *)&aborted))
                break;
            const uint32_t acc = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(a * (int)kTmemCols);
#pragma unroll
            for (int ch = 0; ch < TN / 32; ++ch) {
                uint32_t r[32];
                tmem_ld32(acc + (uint32_t)(ch * 32), r);
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    v[j] = p.alpha * __uint_as_float(r[j]);
                const int col0 = n0 + ch * 32;
                // Mirror of a symmetric product: (col, row) lies in the tile
                // (col / TM, row / TN), not computed when row / TN < col / TM
                // (TM == TN). Uniform over the warp (its rows share row / TN)
                // and the chunk (its columns share col / TM).
                const bool mirror = p.sym && row0 / TN < col0 / TM;
                const bool trans = mirror || p.trans != 0;
                const uint32_t rb = wbuf + (uint32_t)((staged & 1) * kChunkBytes);
                const uint32_t tb = rb + (uint32_t)(2 * kChunkBytes);
                if (lane == 0)   // the buffers' previous group has been read
                    asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                __syncwarp();
                if (crow != nullptr) {
                    // the coalesced chunk of C into rb, then this lane's row out
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const uint4 cv = cpre[ch % kCPre][i];
                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};"
                                     ::"r"(rb + swz64(crs + 8 * i, cg)), "r"(cv.x), "r"(cv.y),
                                       "r"(cv.z), "r"(cv.w)
                                     : "memory");
                        if (ch + kCPre < TN / 32)   // the slot's next chunk
                            cpre[ch % kCPre][i] = __ldg(
                                reinterpret_cast<const uint4 *>(crow + i * c8 + (ch + kCPre) * 32));
                    }
                    __syncwarp();
#pragma unroll
                    for (int g = 0; g < 4; ++g) {
                        uint4 cv;
                        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(cv.x), "=r"(cv.y), "=r"(cv.z), "=r"(cv.w)
                                     : "r"(rb + swz64(lane, g))
                                     : "memory");
                        const __nv_bfloat162 *c2 = reinterpret_cast<const __nv_bfloat162 *>(&cv);
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float2 f = __bfloat1622float2(c2[e]);
                            v[g * 8 + 2 * e] = fmaf(p.beta, f.x, v[g * 8 + 2 * e]);
                            v[g * 8 + 2 * e + 1] = fmaf(p.beta, f.y, v[g * 8 + 2 * e + 1]);
                        }
                    }
                    // each lane rewrites only the row it has read
                }
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const uint32_t w0 = pack_bf16(v[g * 8 + 0], v[g * 8 + 1]);
                    const uint32_t w1 = pack_bf16(v[g * 8 + 2], v[g * 8 + 3]);
                    const uint32_t w2 = pack_bf16(v[g * 8 + 4], v[g * 8 + 5]);
                    const uint32_t w3 = pack_bf16(v[g * 8 + 6], v[g * 8 + 7]);
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(rb + swz64(lane, g)),
                                 "r"(w0), "r"(w1), "r"(w2), "r"(w3)
                                 : "memory");
                }
                if (trans) {   // element (row, col0 + j) at row j, column lane of the transpose
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const __nv_bfloat16 h = __float2bfloat16_rn(v[j]);
                        asm volatile("st.shared.b16 [%0], %1;" ::"r"(tb + swz64(j, lane >> 3) +
                                                                      (uint32_t)((lane & 7) * 2)),
                                     "h"(*reinterpret_cast<const uint16_t *>(&h))
                                     : "memory");
                    }
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) {
                    tma_store_3d(&G.d, rb, col0, row0, b);
                    if (trans)
                        tma_store_3d(mirror ? &G.d : &G.dt, tb, row0, col0, b);
                    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
                }
                ++staged;
            }
            // this warp's rows of the accumulator are read: release them to
            // the leader's MMA lane
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0)
                mbar_arrive_cluster(map_to_rank(acc_empty(a), 0));
            ++lt;
        }
        if (lane == 0)   // every store has been written before the CTA ends
            asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
        __syncwarp();
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    }
    __syncthreads();
    cluster_sync();   // no CTA leaves while its peer may still read its shared memory
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(2 * kTmemCols)
                     : "memory");
    }
}

}  // namespace gemm
}  // namespace dpo
