// aq_store: device storage for one layer that holds only a prefix of its codebooks.
//
// One stored model serves every bit width, and a device holds as many codebooks as its memory
// or latency budget allows (Sec. 1 and Sec. 5). Because the code planes are codebook-major,
// the planes of a prefix m are one contiguous range, so growing the prefix appends planes and
// shrinking it drops a tail. Dropping is ordered on the caller's stream: the dropped
// allocations are released once that stream has passed the call (an event), checked at the
// next call on the store, so no other stream of the process is made to wait.
//
// The store reserves device address space for the whole layer once and backs it with physical
// memory through the CUDA virtual-memory calls (cuMemAddressReserve, cuMemCreate, cuMemMap):
//   [head: scales | codebooks of all M books] [planes 0..M-1]
// The head is mapped when the store is created (the codebooks are small: 2^B*16 bytes per
// book); the plane range is mapped only as far as the resident prefix needs, in whole
// allocation granules. Raising the prefix maps one physical allocation per new plane (the
// granules it does not share with the plane before) and copies the new planes in; lowering it
// releases the allocations that lie wholly past the new prefix. Addresses never move, so pointers into the store stay valid for its life
// (a plain allocation would have to be reallocated and copied to grow).
//
// The driver calls are looked up through the runtime (cudaGetDriverEntryPointByVersion), so
// the library does not link against libcuda.
#include <cuda.h>

#include <mutex>
#include <new>
#include <vector>

#include "aq_internal.cuh"

namespace {

using aq::Dims;

typedef CUresult (*PfnReserve)(CUdeviceptr*, size_t, size_t, CUdeviceptr, unsigned long long);
typedef CUresult (*PfnAddrFree)(CUdeviceptr, size_t);
typedef CUresult (*PfnCreate)(CUmemGenericAllocationHandle*, size_t, const CUmemAllocationProp*,
                              unsigned long long);
typedef CUresult (*PfnRelease)(CUmemGenericAllocationHandle);
typedef CUresult (*PfnMap)(CUdeviceptr, size_t, size_t, CUmemGenericAllocationHandle,
                           unsigned long long);
typedef CUresult (*PfnUnmap)(CUdeviceptr, size_t);
typedef CUresult (*PfnSetAccess)(CUdeviceptr, size_t, const CUmemAccessDesc*, size_t);
typedef CUresult (*PfnGranularity)(size_t*, const CUmemAllocationProp*,
                                   CUmemAllocationGranularity_flags);
typedef CUresult (*PfnErrorName)(CUresult, const char**);

struct Driver {
    PfnReserve reserve;
    PfnAddrFree addr_free;
    PfnCreate create;
    PfnRelease release;
    PfnMap map;
    PfnUnmap unmap;
    PfnSetAccess set_access;
    PfnGranularity granularity;
    PfnErrorName error_name;
};

aq_status lookup(const char* name, void** fn) {
    cudaDriverEntryPointQueryResult q;
    if (cudaError_t e = cudaGetDriverEntryPointByVersion(name, fn, 12000, cudaEnableDefault, &q);
        e != cudaSuccess)
        return aq::cuda_fail(e, "cudaGetDriverEntryPointByVersion");
    if (q != cudaDriverEntryPointSuccess || !*fn) return aq::driver_fail(0, "symbol not found", name);
    return AQ_OK;
}

aq_status driver(const Driver** out) {
    static std::mutex mu;
    static Driver drv;
    static bool have = false;
    std::lock_guard<std::mutex> lock(mu);
    if (!have) {
        void* p[9] = {};
        const char* names[9] = {"cuMemAddressReserve", "cuMemAddressFree", "cuMemCreate",
                                "cuMemRelease", "cuMemMap", "cuMemUnmap", "cuMemSetAccess",
                                "cuMemGetAllocationGranularity", "cuGetErrorName"};
        for (int i = 0; i < 9; ++i)
            if (aq_status e = lookup(names[i], &p[i]); e != AQ_OK) return e;
        drv.reserve = (PfnReserve)p[0];
        drv.addr_free = (PfnAddrFree)p[1];
        drv.create = (PfnCreate)p[2];
        drv.release = (PfnRelease)p[3];
        drv.map = (PfnMap)p[4];
        drv.unmap = (PfnUnmap)p[5];
        drv.set_access = (PfnSetAccess)p[6];
        drv.granularity = (PfnGranularity)p[7];
        drv.error_name = (PfnErrorName)p[8];
        have = true;
    }
    *out = &drv;
    return AQ_OK;
}

aq_status drv_ok(const Driver* drv, CUresult r, const char* what) {
    if (r == CUDA_SUCCESS) return AQ_OK;
    const char* name = nullptr;
    if (drv->error_name(r, &name) != CUDA_SUCCESS) name = nullptr;
    return aq::driver_fail((int)r, name, what);
}

CUmemAllocationProp device_prop(int dev) {
    CUmemAllocationProp prop = {};
    prop.type = CU_MEM_ALLOCATION_TYPE_PINNED;
    prop.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    prop.location.id = dev;
    return prop;
}

// One physical allocation mapped at [addr, addr + bytes).
struct Mapping {
    CUdeviceptr addr;
    size_t bytes;
    CUmemGenericAllocationHandle handle;
};

// Creates a physical allocation of `bytes` (a multiple of the granularity) on dev, maps it at
// addr and makes it readable and writable from dev. On failure nothing stays allocated.
aq_status map_new(const Driver* drv, int dev, CUdeviceptr addr, size_t bytes, Mapping* out) {
    const CUmemAllocationProp prop = device_prop(dev);
    CUmemGenericAllocationHandle h = 0;
    if (aq_status e = drv_ok(drv, drv->create(&h, bytes, &prop, 0), "cuMemCreate"); e != AQ_OK)
        return e;
    if (aq_status e = drv_ok(drv, drv->map(addr, bytes, 0, h, 0), "cuMemMap"); e != AQ_OK) {
        drv->release(h);
        return e;
    }
    CUmemAccessDesc acc = {};
    acc.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    acc.location.id = dev;
    acc.flags = CU_MEM_ACCESS_FLAGS_PROT_READWRITE;
    if (aq_status e = drv_ok(drv, drv->set_access(addr, bytes, &acc, 1), "cuMemSetAccess");
        e != AQ_OK) {
        drv->unmap(addr, bytes);
        drv->release(h);
        return e;
    }
    *out = Mapping{addr, bytes, h};
    return AQ_OK;
}

aq_status unmap_one(const Driver* drv, const Mapping& mp) {
    aq_status e = drv_ok(drv, drv->unmap(mp.addr, mp.bytes), "cuMemUnmap");
    const aq_status e2 = drv_ok(drv, drv->release(mp.handle), "cuMemRelease");
    return e != AQ_OK ? e : e2;
}

// Runs cudaDeviceSynchronize on dev with dev current, then restores the caller's device.
aq_status sync_device(int dev) {
    int cur = 0;
    if (cudaError_t e = cudaGetDevice(&cur); e != cudaSuccess) return aq::cuda_fail(e, "cudaGetDevice");
    if (cur != dev)
        if (cudaError_t e = cudaSetDevice(dev); e != cudaSuccess) return aq::cuda_fail(e, "cudaSetDevice");
    const cudaError_t e = cudaDeviceSynchronize();
    if (cur != dev) cudaSetDevice(cur);
    return aq::cuda_ok(e, "cudaDeviceSynchronize");
}

}  // namespace

// A dropped plane allocation waiting for the work enqueued before its drop to finish.
struct Pending {
    Mapping mp;
    cudaEvent_t done;
};

struct aq_store {
    Dims d;
    int dev;
    size_t gran;                 // allocation granularity of dev
    CUdeviceptr base;            // start of the reserved range
    size_t reserved;             // bytes reserved
    size_t head_bytes;           // scales + codebooks, mapped at creation
    size_t books_off;            // codebooks' offset in the head
    size_t book_bytes;           // one codebook: 2^B codewords of 8 elements
    Mapping head;
    std::vector<Mapping> planes; // mappings of the plane range, in address order
    size_t planes_mapped;        // bytes of the plane range mapped (sum of `planes`)
    std::vector<Pending> pending;  // dropped mappings above the resident ones, in address order
    int m;                       // resident prefix
};

namespace {

CUdeviceptr planes_base(const aq_store* s) { return s->base + s->head_bytes; }

// Unmaps the plane mappings that lie wholly at or past `keep` bytes of the plane range, now.
aq_status drop_planes(const Driver* drv, aq_store* s, size_t keep) {
    aq_status st = AQ_OK;
    while (!s->planes.empty() && s->planes.back().addr >= planes_base(s) + keep) {
        const aq_status e = unmap_one(drv, s->planes.back());
        if (st == AQ_OK) st = e;
        s->planes_mapped -= s->planes.back().bytes;
        s->planes.pop_back();
    }
    return st;
}

// Releases the dropped mappings whose stream work has finished (all of them with wait).
aq_status reap(const Driver* drv, aq_store* s, bool wait) {
    aq_status st = AQ_OK;
    for (size_t i = 0; i < s->pending.size();) {
        Pending& p = s->pending[i];
        const cudaError_t q = wait ? cudaEventSynchronize(p.done) : cudaEventQuery(p.done);
        if (q == cudaErrorNotReady) {
            ++i;
            continue;
        }
        if (q != cudaSuccess && st == AQ_OK) st = aq::cuda_fail(q, "cudaEventQuery");
        const aq_status e = unmap_one(drv, p.mp);
        if (st == AQ_OK) st = e;
        cudaEventDestroy(p.done);
        s->pending.erase(s->pending.begin() + (long)i);
    }
    return st;
}

// Moves the mappings that lie wholly at or past `keep` bytes of the plane range to the pending
// list, each with an event recorded on stream after the work enqueued so far.
aq_status defer_drop(aq_store* s, size_t keep, cudaStream_t stream) {
    std::vector<Pending> moved;
    while (!s->planes.empty() && s->planes.back().addr >= planes_base(s) + keep) {
        cudaEvent_t ev = nullptr;
        if (cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming); e != cudaSuccess)
            return aq::cuda_fail(e, "cudaEventCreateWithFlags");
        if (cudaError_t e = cudaEventRecord(ev, stream); e != cudaSuccess) {
            cudaEventDestroy(ev);
            return aq::cuda_fail(e, "cudaEventRecord");
        }
        moved.push_back(Pending{s->planes.back(), ev});
        s->planes_mapped -= s->planes.back().bytes;
        s->planes.pop_back();
    }
    // keep the pending list in address order: the newly dropped mappings lie below the older
    // pending ones
    s->pending.insert(s->pending.begin(), moved.rbegin(), moved.rend());
    return AQ_OK;
}

void release_all(const Driver* drv, aq_store* s) {
    for (Pending& p : s->pending) {
        unmap_one(drv, p.mp);
        cudaEventDestroy(p.done);
    }
    s->pending.clear();
    drop_planes(drv, s, 0);
    if (s->head.bytes) unmap_one(drv, s->head);
    if (s->base) drv->addr_free(s->base, s->reserved);
}

}  // namespace

extern "C" aq_status aq_store_create(const aq_layout* layout, aq_store** out) {
    if (!out) return AQ_ERR_INVALID_ARG;
    *out = nullptr;
    Dims d;
    if (aq_status e = aq::make_dims(layout, &d); e != AQ_OK) return e;
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return aq::cuda_fail(e, "cudaGetDevice");
    // Makes sure the device's primary context exists before the driver calls.
    if (cudaError_t e = cudaSetDevice(dev); e != cudaSuccess) return aq::cuda_fail(e, "cudaSetDevice");
    const Driver* drv = nullptr;
    if (aq_status e = driver(&drv); e != AQ_OK) return e;

    const CUmemAllocationProp prop = device_prop(dev);
    size_t gran = 0;
    if (aq_status e = drv_ok(drv, drv->granularity(&gran, &prop, CU_MEM_ALLOC_GRANULARITY_MINIMUM),
                             "cuMemGetAllocationGranularity");
        e != AQ_OK)
        return e;
    if (gran == 0) return aq::driver_fail(0, "zero granularity", "cuMemGetAllocationGranularity");

    aq_store* s = new (std::nothrow) aq_store();
    if (!s) return AQ_ERR_CUDA;
    s->d = d;
    s->dev = dev;
    s->gran = gran;
    s->book_bytes = ((size_t)1 << d.B) * 8 * 2;
    s->books_off = aq::round_up((size_t)d.out * 2, 256);
    s->head_bytes = aq::round_up(s->books_off + (size_t)d.M * s->book_bytes, gran);
    // A layer without rows has empty planes; its plane range is still one granule long, so the
    // plane pointer lies inside the reservation.
    const size_t plane_range = aq::round_up((size_t)d.M * d.plane_bytes, gran);
    s->reserved = s->head_bytes + (plane_range ? plane_range : gran);
    aq_status st = drv_ok(drv, drv->reserve(&s->base, s->reserved, gran, 0, 0), "cuMemAddressReserve");
    if (st == AQ_OK) st = map_new(drv, dev, s->base, s->head_bytes, &s->head);
    if (st != AQ_OK) {
        release_all(drv, s);
        delete s;
        return st;
    }
    *out = s;
    return AQ_OK;
}

extern "C" aq_status aq_store_set_prefix(aq_store* s, int m, const void* src_planes,
                                         const void* src_books, const void* src_scales,
                                         void* stream) {
    if (!s || m < 0 || m > s->d.M) return AQ_ERR_INVALID_ARG;
    const int m0 = s->m;
    if (m == m0) return AQ_OK;
    if (m > m0 && (!src_planes || !src_books || (m0 == 0 && !src_scales))) return AQ_ERR_INVALID_ARG;
    const Driver* drv = nullptr;
    if (aq_status e = driver(&drv); e != AQ_OK) return e;
    const size_t pb = s->d.plane_bytes;

    const cudaStream_t st = (cudaStream_t)stream;
    // dropped allocations whose stream work has finished are released now
    const aq_status reaped = reap(drv, s, false);
    if (m < m0) {
        // The memory of the dropped planes is released once `stream` has passed this point
        // (work reading them must be ordered before the call on it); other streams run on.
        const aq_status e = defer_drop(s, aq::round_up((size_t)m * pb, s->gran), st);
        s->m = m;
        return e != AQ_OK ? e : reaped;
    }

    const size_t need = aq::round_up((size_t)m * pb, s->gran);
    // Dropped allocations still waiting for their release lie right where the planes grow:
    // take them back (their addresses cannot be mapped twice; their contents are rewritten by
    // the copies below).
    while (need > s->planes_mapped && !s->pending.empty() &&
           s->pending.front().mp.addr == planes_base(s) + s->planes_mapped) {
        s->planes.push_back(s->pending.front().mp);
        s->planes_mapped += s->pending.front().mp.bytes;
        cudaEventDestroy(s->pending.front().done);
        s->pending.erase(s->pending.begin());
    }
    // One allocation per plane (its granules not yet mapped), so that lowering later can give
    // back every plane it drops.
    for (int k = m0; k < m && need > s->planes_mapped; ++k) {
        const size_t end = aq::round_up((size_t)(k + 1) * pb, s->gran);
        if (end <= s->planes_mapped) continue;
        Mapping mp;
        if (aq_status e = map_new(drv, s->dev, planes_base(s) + s->planes_mapped,
                                  end - s->planes_mapped, &mp);
            e != AQ_OK)
            return e;
        s->planes.push_back(mp);
        s->planes_mapped = end;
    }
    unsigned char* dst = (unsigned char*)s->base;
    const size_t off = (size_t)m0 * pb, n = (size_t)(m - m0) * pb;
    if (n)
        if (aq_status e = aq::cuda_ok(cudaMemcpyAsync(dst + s->head_bytes + off,
                                                      (const unsigned char*)src_planes + off, n,
                                                      cudaMemcpyDefault, st),
                                      "cudaMemcpyAsync (planes)");
            e != AQ_OK)
            return e;
    const size_t boff = (size_t)m0 * s->book_bytes, bn = (size_t)(m - m0) * s->book_bytes;
    if (aq_status e = aq::cuda_ok(cudaMemcpyAsync(dst + s->books_off + boff,
                                                  (const unsigned char*)src_books + boff, bn,
                                                  cudaMemcpyDefault, st),
                                  "cudaMemcpyAsync (codebooks)");
        e != AQ_OK)
        return e;
    if (m0 == 0 && s->d.out > 0)
        if (aq_status e = aq::cuda_ok(cudaMemcpyAsync(dst, src_scales, (size_t)s->d.out * 2,
                                                      cudaMemcpyDefault, st),
                                      "cudaMemcpyAsync (scales)");
            e != AQ_OK)
            return e;
    s->m = m;
    return AQ_OK;
}

extern "C" int aq_store_prefix(const aq_store* s) { return s ? s->m : 0; }

extern "C" void* aq_store_planes(const aq_store* s) {
    return s ? (void*)(s->base + s->head_bytes) : nullptr;
}

extern "C" void* aq_store_books(const aq_store* s) {
    return s ? (void*)(s->base + s->books_off) : nullptr;
}

extern "C" void* aq_store_scales(const aq_store* s) { return s ? (void*)s->base : nullptr; }

extern "C" size_t aq_store_device_bytes(aq_store* s) {
    if (!s) return 0;
    const Driver* drv = nullptr;
    if (driver(&drv) == AQ_OK) reap(drv, s, false);
    size_t held = s->head_bytes + s->planes_mapped;
    for (const Pending& p : s->pending) held += p.mp.bytes;
    return held;
}

extern "C" aq_status aq_store_destroy(aq_store* s) {
    if (!s) return AQ_OK;
    const Driver* drv = nullptr;
    if (aq_status e = driver(&drv); e != AQ_OK) return e;
    const aq_status e = sync_device(s->dev);
    release_all(drv, s);
    delete s;
    return e;
}
