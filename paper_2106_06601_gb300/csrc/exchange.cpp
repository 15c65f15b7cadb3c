// Multi-GPU exchange of COSTA's reshuffle A = alpha * op(B) + beta * A
// (Sec. 6 "Implementation", Alg. 3), with the P ranks placed on G GPUs.
//
// Alg. 3 has every process pack its outgoing packages, send them, and
// transform each package into A as it arrives; blocks that stay on their
// process skip the buffers.  Here the process is a GPU: rank r's blocks live
// on GPU place[r], and GPU g runs
//   pack   - the tiles whose source rank is on g and whose target rank is on
//            another GPU h, copied exactly (the transform comes after the
//            transfer) into h's segment of g's send buffer;
//   local  - the tiles whose source and target ranks are both on g, straight
//            from B to A (the direct remap);
//   unpack - the tiles received from each GPU h, from h's segment of g's
//            receive buffer into A, with op, alpha and beta.
// Between pack and unpack the caller moves every send segment to its
// receiver (one all-to-all-v, e.g. NCCL's grouped send/receive); the
// library itself never touches another GPU's memory.
//
// No coordination is needed to agree on the packages: each GPU cuts the
// same tiles from the layouts (the overlay depends only on splits and
// storage orders, not on pointers) and enumerates them in one canonical
// order, fixed here and independent of any tuning override.  A package
// (g -> h) holds, in that order, the tiles with source on g and target on
// h, each dense in the source's element order with its leading dimension
// rounded up to 16 bytes; its tiles' offsets are the running sums of their
// sizes, which sender and receiver compute alike.  Segments are ordered by
// peer at the exclusive-scan offsets of the package sizes (all-to-all-v
// displacements).
#include <cuda_runtime_api.h>

#include <cstdio>
#include <cstring>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "costa_internal.h"
#include "plan_lists.h"
#include "tiles.h"

struct costa_exchange_s {
    int device = 0;
    int G = 1, g = 0;
    int dtype = 0, esize = 0;
    std::vector<int64_t> send_bytes, recv_bytes;
    void *d_mem = nullptr;
    costa::DevList pack, local, unpack, local_halves, unpack_halves;
    ~costa_exchange_s() {
        if (d_mem) cudaFree(d_mem);
    }
};

namespace costa {

costa_status fail_msg(costa_status s, const std::string &m) { return report_error(s, m.c_str()); }
costa_status cuda_msg(cudaError_t e, const char *what) {
    return fail_msg(COSTA_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

struct ExchangeLists {
    std::vector<TileDesc> pack, local, unpack;
    std::vector<int64_t> send_elems, recv_elems;  // per peer GPU, elements of the packed tiles
    std::vector<int64_t> send_volume, recv_volume;  // per peer GPU, elements of A moved
};

costa_status check_placement(int P, int G, const int *place, int g) {
    if (G < 1) return fail_msg(COSTA_ERR_INVALID_ARG, "G = " + std::to_string(G) + " < 1");
    if (g < 0 || g >= G) return fail_msg(COSTA_ERR_INVALID_ARG, "GPU index out of [0, G)");
    if (!place) return fail_msg(COSTA_ERR_INVALID_ARG, "place is null");
    for (int r = 0; r < P; ++r)
        if (place[r] < 0 || place[r] >= G)
            return fail_msg(COSTA_ERR_INVALID_ARG,
                            "place[" + std::to_string(r) + "] = " + std::to_string(place[r]) + " not in [0, G)");
    return COSTA_OK;
}

// The canonical tile order of the exchange: super-tiles of k x k pieces
// (k = 16 for 16-byte elements, 8 otherwise), row pieces fastest.
template <typename F> void exchange_tile_order(const ProblemHost &ph, F &&f) {
    const int k = esize_of(ph.A->dt) == 16 ? 16 : 8;
    const int nu = static_cast<int>(ph.rows.tiles.size()), nv = static_cast<int>(ph.cols.tiles.size());
    for (int su = 0; su < nu; su += k)
        for (int sv = 0; sv < nv; sv += k)
            for (int v = sv; v < std::min(sv + k, nv); ++v)
                for (int u = su; u < std::min(su + k, nu); ++u) f(ph.rows.tiles[u], ph.cols.tiles[v]);
}

// The three tile lists of GPU g (see the file comment).  send_base and
// recv_base are the addresses of g's send and receive buffers.
costa_status plan_exchange(const costa_layout_s *A, const costa_layout_s *B, int op, int G, const int *place,
                           int g, uint64_t send_base, uint64_t recv_base, ExchangeLists &out) {
    costa_status s = check_pair(A, B, op);
    if (s != COSTA_OK) return s;
    s = check_placement(A->nranks, G, place, g);
    if (s != COSTA_OK) return s;
    const int es = esize_of(A->dt), ts = tile_extent(es), vec = 16 / es;
    ProblemHost ph;
    ph.A = A;
    ph.B = B;
    ph.op = static_cast<costa_op>(op);
    ph.rows = cut_pair_axis(A, B, op, 0, ts);
    ph.cols = cut_pair_axis(A, B, op, 1, ts);
    const bool tr = op != COSTA_OP_N;
    struct Remote {
        TileDesc d;
        int peer;
        int32_t ld;
        int64_t off;  // elements from the start of the package
    };
    std::vector<Remote> sends, recvs;
    out = ExchangeLists{};
    out.send_elems.assign(G, 0);
    out.recv_elems.assign(G, 0);
    out.send_volume.assign(G, 0);
    out.recv_volume.assign(G, 0);
    exchange_tile_order(ph, [&](const AxisTile &rt, const AxisTile &ct) {
        const int q = A->owner[static_cast<size_t>(rt.a_blk) * A->nbc + ct.a_blk];
        const size_t bidx = tr ? static_cast<size_t>(ct.b_blk) * B->nbc + rt.b_blk
                               : static_cast<size_t>(rt.b_blk) * B->nbc + ct.b_blk;
        const int p = B->owner[bidx];
        const int gp = place[p], gq = place[q];
        if (gp != g && gq != g) return;
        TileDesc d = direct_tile(ph, rt, ct, es, 0);
        if (gp == g && gq == g) {
            set_fast(d, es);
            out.local.push_back(d);
            return;
        }
        const bool t = (d.flags & TF_TRANSPOSE) != 0;
        const int fast = t ? d.ny : d.nx, other = t ? d.nx : d.ny;  // source frame
        Remote r;
        r.d = d;
        r.ld = (fast + vec - 1) / vec * vec;
        const int64_t size = static_cast<int64_t>(r.ld) * other;
        if (gp == g) {
            r.peer = gq;
            r.off = out.send_elems[gq];
            out.send_elems[gq] += size;
            out.send_volume[gq] += static_cast<int64_t>(d.nx) * d.ny;
            sends.push_back(r);
        } else {
            r.peer = gp;
            r.off = out.recv_elems[gp];
            out.recv_elems[gp] += size;
            out.recv_volume[gp] += static_cast<int64_t>(d.nx) * d.ny;
            recvs.push_back(r);
        }
    });
    std::vector<int64_t> sdispl(G, 0), rdispl(G, 0);
    for (int h = 1; h < G; ++h) {
        sdispl[h] = sdispl[h - 1] + out.send_elems[h - 1];
        rdispl[h] = rdispl[h - 1] + out.recv_elems[h - 1];
    }
    out.pack.reserve(sends.size());
    for (const Remote &r : sends) {  // an exact copy in the source's frame
        TileDesc pk = r.d;
        const bool t = (r.d.flags & TF_TRANSPOSE) != 0;
        pk.nx = t ? r.d.ny : r.d.nx;
        pk.ny = t ? r.d.nx : r.d.ny;
        pk.dst = send_base + static_cast<uint64_t>((sdispl[r.peer] + r.off) * es);
        pk.dld = r.ld;
        pk.flags = 0;
        set_fast(pk, es);
        out.pack.push_back(pk);
    }
    out.unpack.reserve(recvs.size());
    for (const Remote &r : recvs) {  // the direct tile, reading the received copy
        TileDesc up = r.d;
        up.src = recv_base + static_cast<uint64_t>((rdispl[r.peer] + r.off) * es);
        up.sld = r.ld;
        set_fast(up, es);
        out.unpack.push_back(up);
    }
    for (const auto &l : {std::make_pair(&out.pack, "pack"), std::make_pair(&out.local, "local"),
                          std::make_pair(&out.unpack, "unpack")}) {
        s = check_extents(*l.first, es, l.second);
        if (s != COSTA_OK) return s;
    }
    // The lists that write A take the direct path's order in the target's
    // own storage where that one does (the offsets above are fixed already,
    // so this changes only which tiles are in flight together).
    if (use_local_order(ph, out.local.data(), out.local.size()))
        for (std::vector<TileDesc> *l : {&out.local, &out.unpack}) {
            bool contiguous = true;
            for (size_t i = 0; i < l->size() && contiguous; ++i) contiguous = (*l)[i].nx == (*l)[i].dld;
            if (!contiguous) order_tiles_local(*l, 0, l->size(), es, ts);
        }
    return COSTA_OK;
}

bool device_buffer_ok(const void *p, int dev) {
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return (at.type == cudaMemoryTypeDevice && at.device == dev) || at.type == cudaMemoryTypeManaged;
}

costa_status exchange_launch(costa_exchange_s *x, const DevList &list, const DevList *halves, const void *alpha,
                             const void *beta, void *stream_v, bool copy) {
    if (!x) return fail_msg(COSTA_ERR_INVALID_ARG, "null exchange");
    if (!copy && (!alpha || !beta)) return fail_msg(COSTA_ERR_INVALID_ARG, "null scalar");
    if (list.empty()) return COSTA_OK;
    int dev = 0;
    cudaError_t ce = cudaGetDevice(&dev);
    if (ce != cudaSuccess) return cuda_msg(ce, "cudaGetDevice");
    if (dev != x->device)
        return fail_msg(COSTA_ERR_INVALID_ARG, "the current device is not the exchange's device");
    RemapLaunch L{};
    L.dtype = x->dtype;
    L.per_problem = nullptr;
    bool kinds[K_NKINDS] = {};
    if (copy) {
        const float one_f[2] = {1.0f, 0.0f}, zero_f[2] = {0.0f, 0.0f};
        const double one_d[2] = {1.0, 0.0}, zero_d[2] = {0.0, 0.0};
        const bool single = x->dtype == COSTA_F32 || x->dtype == COSTA_C64;
        L.s = make_scalars(x->dtype, single ? static_cast<const void *>(one_f) : one_d,
                           single ? static_cast<const void *>(zero_f) : zero_d, 0);
        kinds[K_COPY] = true;
    } else {
        L.s = make_scalars(x->dtype, alpha, beta, 0);
        kinds[kind_of(L.s.flags)] = true;
    }
    ce = launch_split(L, list, halves, x->esize, kinds, static_cast<cudaStream_t>(stream_v));
    if (ce != cudaSuccess) return cuda_msg(ce, "exchange kernel launch");
    return COSTA_OK;
}

}  // namespace costa

using namespace costa;

extern "C" {

costa_status costa_exchange_sizes(costa_layout A, costa_layout B, costa_op op, int G, const int *place, int g,
                                  int64_t *send_bytes, int64_t *recv_bytes) {
    if (!send_bytes || !recv_bytes) return fail_msg(COSTA_ERR_INVALID_ARG, "null output");
    ExchangeLists l;
    costa_status s = plan_exchange(A, B, op, G, place, g, 0, 0, l);
    if (s != COSTA_OK) return s;
    const int es = esize_of(A->dt);
    for (int h = 0; h < G; ++h) {
        send_bytes[h] = l.send_elems[h] * es;
        recv_bytes[h] = l.recv_elems[h] * es;
    }
    return COSTA_OK;
}

costa_status costa_exchange_create(costa_exchange *out, costa_layout A, costa_layout B, costa_op op, int G,
                                   const int *place, int g, void *send_buf, void *recv_buf) {
    if (!out) return fail_msg(COSTA_ERR_INVALID_ARG, "out is null");
    *out = nullptr;
    Trace trace("costa exchange plan");
    auto x = std::make_unique<costa_exchange_s>();
    cudaError_t ce = cudaGetDevice(&x->device);
    if (ce != cudaSuccess) return cuda_msg(ce, "cudaGetDevice");
    ExchangeLists l;
    costa_status s = plan_exchange(A, B, op, G, place, g, reinterpret_cast<uint64_t>(send_buf),
                                   reinterpret_cast<uint64_t>(recv_buf), l);
    if (s != COSTA_OK) return s;
    s = check_access_on(A, x->device, "A", place, g);
    if (s == COSTA_OK) s = check_access_on(B, x->device, "B", place, g);
    if (s != COSTA_OK) return s;
    const int es = esize_of(A->dt);
    int64_t nsend = 0, nrecv = 0;
    for (int h = 0; h < G; ++h) {
        nsend += l.send_elems[h];
        nrecv += l.recv_elems[h];
    }
    if (nsend > 0 && (!send_buf || !device_buffer_ok(send_buf, x->device) ||
                      !device_buffer_ok(static_cast<char *>(send_buf) + nsend * es - 1, x->device)))
        return fail_msg(COSTA_ERR_INVALID_ARG, "send buffer is not device memory of " +
                                                   std::to_string(nsend * es) + " bytes on the current device");
    if (nrecv > 0 && (!recv_buf || !device_buffer_ok(recv_buf, x->device) ||
                      !device_buffer_ok(static_cast<char *>(recv_buf) + nrecv * es - 1, x->device)))
        return fail_msg(COSTA_ERR_INVALID_ARG, "receive buffer is not device memory of " +
                                                   std::to_string(nrecv * es) + " bytes on the current device");
    if ((nsend > 0 && reinterpret_cast<uintptr_t>(send_buf) % 16) ||
        (nrecv > 0 && reinterpret_cast<uintptr_t>(recv_buf) % 16))
        return fail_msg(COSTA_ERR_INVALID_ARG, "send and receive buffers must be 16-byte aligned");
    x->G = G;
    x->g = g;
    x->dtype = A->dt;
    x->esize = es;
    x->send_bytes.resize(G);
    x->recv_bytes.resize(G);
    for (int h = 0; h < G; ++h) {
        x->send_bytes[h] = l.send_elems[h] * es;
        x->recv_bytes[h] = l.recv_elems[h] * es;
    }
    const bool cplx = A->dt == COSTA_C64 || A->dt == COSTA_C128;
    const SplitList s_pack = split_small(std::move(l.pack), es, cplx),
                    s_local = split_small(std::move(l.local), es, cplx),
                    s_unpack = split_small(std::move(l.unpack), es, cplx);
    ProblemHost ph;
    ph.A = A;
    ph.B = B;
    ph.op = op;
    const std::vector<char> halve(1, use_halves(ph, es) ? 1 : 0);
    const std::vector<TileDesc> h_local = split_x_halves(s_local.big, tile_extent(es) / 2, es, halve),
                                h_unpack = split_x_halves(s_unpack.big, tile_extent(es) / 2, es, halve);
    Arena arena;
    const SplitOffsets o_pack = arena.add_split(s_pack);
    const SplitOffsets o_local = arena.add_split(s_local);
    const SplitOffsets o_unpack = arena.add_split(s_unpack);
    const size_t o_hl = h_local.empty() ? 0 : arena.add_vec(h_local);
    const size_t o_hu = h_unpack.empty() ? 0 : arena.add_vec(h_unpack);
    ce = cudaMalloc(&x->d_mem, arena.host.size());
    if (ce != cudaSuccess) {
        x->d_mem = nullptr;
        return fail_msg(COSTA_ERR_ALLOC, std::string("cudaMalloc(exchange tables): ") + cudaGetErrorString(ce));
    }
    ce = cudaMemcpy(x->d_mem, arena.host.data(), arena.host.size(), cudaMemcpyHostToDevice);
    if (ce != cudaSuccess) return cuda_msg(ce, "cudaMemcpy(exchange tables)");
    const char *db = static_cast<const char *>(x->d_mem);
    x->pack = resolve(db, o_pack, s_pack);
    x->local = resolve(db, o_local, s_local);
    x->unpack = resolve(db, o_unpack, s_unpack);
    x->local_halves = x->local;
    x->unpack_halves = x->unpack;
    if (!h_local.empty()) {
        x->local_halves.tiles = reinterpret_cast<const TileDesc *>(db + o_hl);
        x->local_halves.ntiles = static_cast<int64_t>(h_local.size());
    }
    if (!h_unpack.empty()) {
        x->unpack_halves.tiles = reinterpret_cast<const TileDesc *>(db + o_hu);
        x->unpack_halves.ntiles = static_cast<int64_t>(h_unpack.size());
    }
    log_msg(1, "exchange plan: GPU %d of %d, send %lld bytes, receive %lld bytes; pack %zu, local %zu, "
               "unpack %zu tiles", g, G, (long long)(nsend * es), (long long)(nrecv * es),
            s_pack.big.size() + s_pack.mis.size() + s_pack.pieces.size(),
            s_local.big.size() + s_local.mis.size() + s_local.pieces.size(),
            s_unpack.big.size() + s_unpack.mis.size() + s_unpack.pieces.size());
    *out = x.release();
    return COSTA_OK;
}

costa_status costa_exchange_counts(costa_exchange x, int64_t *send_bytes, int64_t *recv_bytes) {
    if (!x || !send_bytes || !recv_bytes) return fail_msg(COSTA_ERR_INVALID_ARG, "null argument");
    for (int h = 0; h < x->G; ++h) {
        send_bytes[h] = x->send_bytes[h];
        recv_bytes[h] = x->recv_bytes[h];
    }
    return COSTA_OK;
}

costa_status costa_exchange_pack(costa_exchange x, void *stream) {
    Trace trace("costa exchange pack");
    if (!x) return fail_msg(COSTA_ERR_INVALID_ARG, "null exchange");
    return exchange_launch(x, x->pack, nullptr, nullptr, nullptr, stream, true);
}

costa_status costa_exchange_local(costa_exchange x, const void *alpha, const void *beta, void *stream) {
    Trace trace("costa exchange local");
    if (!x) return fail_msg(COSTA_ERR_INVALID_ARG, "null exchange");
    return exchange_launch(x, x->local, &x->local_halves, alpha, beta, stream, false);
}

costa_status costa_exchange_unpack(costa_exchange x, const void *alpha, const void *beta, void *stream) {
    Trace trace("costa exchange unpack");
    if (!x) return fail_msg(COSTA_ERR_INVALID_ARG, "null exchange");
    return exchange_launch(x, x->unpack, &x->unpack_halves, alpha, beta, stream, false);
}

costa_status costa_exchange_destroy(costa_exchange x) {
    delete x;
    return COSTA_OK;
}

costa_status costa_debug_exchange(costa_layout A, costa_layout B, costa_op op, int G, const int *place, int g,
                                  uint64_t send_base, uint64_t recv_base, int which, void *out, int64_t cap,
                                  int64_t *count, int64_t *volumes) {
    if (!count) return fail_msg(COSTA_ERR_INVALID_ARG, "count is null");
    if (which < 0 || which > 2) return fail_msg(COSTA_ERR_INVALID_ARG, "which must be 0, 1 or 2");
    ExchangeLists l;
    costa_status s = plan_exchange(A, B, op, G, place, g, send_base, recv_base, l);
    if (s != COSTA_OK) return s;
    const std::vector<TileDesc> &v = which == 0 ? l.pack : which == 1 ? l.local : l.unpack;
    *count = static_cast<int64_t>(v.size());
    if (out && cap > 0)
        std::memcpy(out, v.data(), sizeof(TileDesc) * static_cast<size_t>(std::min<int64_t>(cap, *count)));
    if (volumes)
        for (int h = 0; h < G; ++h) {
            volumes[h] = l.send_volume[h];
            volumes[G + h] = l.recv_volume[h];
        }
    return COSTA_OK;
}

}  // extern "C"
