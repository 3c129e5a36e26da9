// rlm_iocap.cu -- the memory ceiling of the prefill's access pattern.
//
// The tensor-core prefill gives each CTA one group of 8 channels, so every token
// row it reads or writes is a 16-byte slice of a [B][L][D] row.  This kernel
// streams the same pattern with nothing else in the way: each CTA owns one
// slice (slice_bytes wide) of a [rows][D] bf16 field and a range of its rows,
// loads 4 KB boxes of it with TMA (two producer rings of 8 boxes) and stores the
// same number of 4 KB boxes of the destination field with TMA (up to four bulk
// groups in flight).  Timing it with the prefill's CTA count gives the ceiling
// the prefill can reach for its byte count; comparing slice widths shows what
// the row width costs.
//
// Every wait is bounded (about 2 s); an expired wait ends that role's loop, the CTA
// drains what it issued and returns, and the measured time (seconds instead of
// microseconds) shows it.
#include <cuda.h>

#include <mutex>

#include "rlm_internal.h"

namespace rlm {

namespace {

constexpr int kRing = 8;
constexpr int kProducers = 2;
constexpr int kStoreSlots = 4;
constexpr int kBoxBytes = 4096;
constexpr long long kLimit = 4000000000ll;
constexpr int kIoThreads = 32 * (2 * kProducers + 1);
constexpr int kIoSmem = (kProducers * kRing + kStoreSlots) * kBoxBytes + 2 * kProducers * kRing * 8 + 1024;

__device__ __forceinline__ uint32_t s32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ bool poll(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!poll(bar, parity))
        if (clock64() - t0 > kLimit) return false;
    return true;
}

// boxes: 4 KB boxes each CTA loads (and stores).  Box i of CTA k covers rows
// [r, r + box_rows) of slice (k % slices), r = ((k / slices) * boxes + i) * box_rows
// modulo the field.
__global__ void __launch_bounds__(kIoThreads, 1)
    k_row_io(const __grid_constant__ CUtensorMap src, const __grid_constant__ CUtensorMap dst,
             int64_t rows, int slices, int slice_ch, int box_rows, int boxes) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = smem_raw + ((1024u - (s32(smem_raw) & 1023u)) & 1023u);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (kProducers * kRing + kStoreSlots) * kBoxBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 2 * kProducers * kRing; ++i)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(s32(bars + i)));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    const int ch0 = (blockIdx.x % slices) * slice_ch;
    const int64_t nblocks = rows / box_rows;
    const int64_t first = (int64_t)(blockIdx.x / slices) * boxes;
    const int per = boxes / kProducers;
    if (warp < kProducers && lane == 0) {
        const int p = warp;
        int i = 0;
        for (; i < per; ++i) {
            const int slot = i % kRing, fill = i / kRing;
            const uint32_t full = s32(bars + p * kRing + slot);
            const uint32_t empty = s32(bars + (kProducers + p) * kRing + slot);
            if (!wait_bounded(empty, (fill & 1) ^ 1)) break;
            const int64_t rb = (first + (int64_t)p * per + i) % nblocks;
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(full), "r"(kBoxBytes)
                         : "memory");
            asm volatile(
                "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
                " [%0], [%1, {%2, %3}], [%4];" ::"r"(s32(smem + (p * kRing + slot) * kBoxBytes)),
                "l"(reinterpret_cast<uint64_t>(&src)), "r"(ch0), "r"((int)(rb * box_rows)), "r"(full)
                : "memory");
        }
        // Drain: the last issued loads land before the CTA leaves.
        for (int k = i > kRing ? i - kRing : 0; k < i; ++k)
            wait_bounded(s32(bars + p * kRing + k % kRing), (k / kRing) & 1);
    } else if (warp >= kProducers && warp < 2 * kProducers && lane == 0) {
        const int p = warp - kProducers;
        for (int i = 0; i < per; ++i) {
            const int slot = i % kRing, fill = i / kRing;
            if (!wait_bounded(s32(bars + p * kRing + slot), fill & 1)) break;
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(s32(bars + (kProducers + p) * kRing + slot))
                         : "memory");
        }
    } else if (warp == 2 * kProducers && lane == 0) {
        const uint32_t sb = s32(smem + kProducers * kRing * kBoxBytes);
        for (int i = 0; i < boxes; ++i) {
            const int64_t rb = (first + i) % nblocks;
            asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                             reinterpret_cast<uint64_t>(&dst)),
                         "r"(ch0), "r"((int)(rb * box_rows)), "r"(sb + (i % kStoreSlots) * kBoxBytes)
                         : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(kStoreSlots - 1) : "memory");
        }
        asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    }
    __syncthreads();
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encoder() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

bool field_map(CUtensorMap *map, const void *ptr, int64_t rows, int D, int slice_ch, int box_rows) {
    EncodeTiledFn fn = encoder();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    cuuint32_t box[2] = {(cuuint32_t)slice_ch, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace
}  // namespace rlm

using namespace rlm;

extern "C" rlm_status rlm_measure_row_io(const void *src, void *dst, int64_t rows, int D, int slice_bytes,
                                         int ctas, void *stream) {
    if (!src || !dst) {
        set_error("rlm_measure_row_io: src or dst is NULL");
        return RLM_ERR_INVALID_ARG;
    }
    if ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) {
        set_error("rlm_measure_row_io: src and dst must be 16-byte aligned");
        return RLM_ERR_INVALID_ARG;
    }
    if (slice_bytes != 16 && slice_bytes != 32 && slice_bytes != 64 && slice_bytes != 128) {
        set_error("rlm_measure_row_io: slice_bytes must be 16, 32, 64 or 128");
        return RLM_ERR_INVALID_ARG;
    }
    const int slice_ch = slice_bytes / 2, box_rows = kBoxBytes / slice_bytes;
    if (D < slice_ch || D % slice_ch != 0 || D > (1 << 16)) {
        set_error("rlm_measure_row_io: D must be a multiple of slice_bytes / 2 (and <= 65536)");
        return RLM_ERR_INVALID_ARG;
    }
    const int slices = D / slice_ch;
    if (ctas < 1 || ctas % slices != 0 || ctas > 65535) {
        set_error("rlm_measure_row_io: ctas must be a positive multiple of D / (slice_bytes / 2)");
        return RLM_ERR_INVALID_ARG;
    }
    if (rows < box_rows || rows % box_rows != 0 || rows > INT32_MAX) {
        set_error("rlm_measure_row_io: rows must be a multiple of 4096 / slice_bytes (and < 2^31)");
        return RLM_ERR_INVALID_ARG;
    }
    // Every CTA moves the same number of boxes; together they cover the field once.
    const int64_t total = rows / box_rows * slices;
    int boxes = (int)(total / ctas);
    boxes -= boxes % kProducers;
    if (boxes < kProducers) {
        set_error("rlm_measure_row_io: field too small for %d CTAs", ctas);
        return RLM_ERR_INVALID_ARG;
    }
    CUtensorMap ms, md;
    if (!field_map(&ms, src, rows, D, slice_ch, box_rows) || !field_map(&md, dst, rows, D, slice_ch, box_rows)) {
        set_error("rlm_measure_row_io: tensor map encoding failed");
        return RLM_ERR_CUDA;
    }
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [] {
        attr_err = cudaFuncSetAttribute(k_row_io, cudaFuncAttributeMaxDynamicSharedMemorySize, kIoSmem);
    });
    if (attr_err != cudaSuccess) {
        set_error("rlm_measure_row_io: %s", cudaGetErrorString(attr_err));
        return RLM_ERR_CUDA;
    }
    k_row_io<<<ctas, kIoThreads, kIoSmem, static_cast<cudaStream_t>(stream)>>>(ms, md, rows, slices, slice_ch,
                                                                               box_rows, boxes);
    count_launches(1);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("rlm_measure_row_io launch: %s", cudaGetErrorString(e));
        return RLM_ERR_CUDA;
    }
    return RLM_OK;
}

extern "C" int64_t rlm_measure_row_io_bytes(int64_t rows, int D, int slice_bytes, int ctas) {
    if (slice_bytes <= 0 || ctas <= 0) return 0;
    const int slice_ch = slice_bytes / 2, box_rows = kBoxBytes / slice_bytes;
    if (slice_ch <= 0 || D % slice_ch != 0 || box_rows <= 0) return 0;
    const int64_t total = rows / box_rows * (D / slice_ch);
    int64_t boxes = total / ctas;
    boxes -= boxes % kProducers;
    return 2 * boxes * ctas * kBoxBytes;  // loaded plus stored
}
