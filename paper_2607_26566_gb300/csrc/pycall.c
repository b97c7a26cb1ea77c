/*
 * pycall.c -- CPython entry points for the store's per-request calls.
 *
 * The ctypes binding converts every argument of every call through ctypes'
 * type machinery and releases and re-takes the interpreter lock around it:
 * about 1.5 us per call on a Grace host, as much as a call of the library
 * itself on a small request. This module passes the same arguments (plain
 * integers: the store handle, descriptor and id array addresses, counts and
 * the cudaStream_t) to the same C-ABI functions of libt2istore.so with
 * METH_FASTCALL, and keeps the interpreter lock for the call: a few
 * microseconds of host work, unless the call waits for the store's own lock
 * (another thread is inside the store) or for room in a full launch queue,
 * during which other Python threads wait too (the ctypes binding releases
 * the lock instead). Marshalling only: every check, page table step and
 * byte move happens in the library.
 */
#define PY_SSIZE_T_CLEAN
#include <Python.h>
#include <stdint.h>

#include "t2istore.h"

/* Integer argument i as an address (0 -> NULL). 0 on a Python error. */
static int arg_ptr(PyObject* const* args, Py_ssize_t i, void** out) {
    *out = PyLong_AsVoidPtr(args[i]);
    return !(*out == NULL && PyErr_Occurred());
}

static int arg_u32(PyObject* const* args, Py_ssize_t i, uint32_t* out) {
    const unsigned long v = PyLong_AsUnsignedLong(args[i]);
    if (v == (unsigned long)-1 && PyErr_Occurred()) return 0;
    if (v > 0xFFFFFFFFul) {
        PyErr_SetString(PyExc_OverflowError, "count does not fit uint32");
        return 0;
    }
    *out = (uint32_t)v;
    return 1;
}

static int nargs_ok(Py_ssize_t n, Py_ssize_t want, const char* name) {
    if (n == want) return 1;
    PyErr_Format(PyExc_TypeError, "%s takes %zd arguments (%zd given)", name, want, n);
    return 0;
}

/* put_batch(store, descs, n, out_ids, stream) -> status (t2i_put_batch) */
static PyObject* py_put_batch(PyObject* self, PyObject* const* args, Py_ssize_t n) {
    void *h, *d, *ids, *s;
    uint32_t cnt;
    (void)self;
    if (!nargs_ok(n, 5, "put_batch") || !arg_ptr(args, 0, &h) || !arg_ptr(args, 1, &d) || !arg_u32(args, 2, &cnt) ||
        !arg_ptr(args, 3, &ids) || !arg_ptr(args, 4, &s))
        return NULL;
    return PyLong_FromLong(t2i_put_batch((t2i_store*)h, (const t2i_put_desc*)d, cnt, (t2i_id*)ids, s));
}

/* get_batch(store, descs, n, per_item, stream) -> status (t2i_get_batch;
 * per_item may be 0) */
static PyObject* py_get_batch(PyObject* self, PyObject* const* args, Py_ssize_t n) {
    void *h, *d, *per, *s;
    uint32_t cnt;
    (void)self;
    if (!nargs_ok(n, 5, "get_batch") || !arg_ptr(args, 0, &h) || !arg_ptr(args, 1, &d) || !arg_u32(args, 2, &cnt) ||
        !arg_ptr(args, 3, &per) || !arg_ptr(args, 4, &s))
        return NULL;
    return PyLong_FromLong(t2i_get_batch((t2i_store*)h, (const t2i_get_desc*)d, cnt, (t2i_status*)per, s));
}

/* get_batch_ids(store, descs, n, ids, per_item, stream) -> status: writes
 * ids[0..n) into the id fields of descs[0..n) (a prepared batch whose
 * buffers stay the same, fed with the ids of the put that made its objects),
 * then t2i_get_batch. */
static PyObject* py_get_batch_ids(PyObject* self, PyObject* const* args, Py_ssize_t n) {
    void *h, *d, *ids, *per, *s;
    uint32_t cnt;
    (void)self;
    if (!nargs_ok(n, 6, "get_batch_ids") || !arg_ptr(args, 0, &h) || !arg_ptr(args, 1, &d) ||
        !arg_u32(args, 2, &cnt) || !arg_ptr(args, 3, &ids) || !arg_ptr(args, 4, &per) || !arg_ptr(args, 5, &s))
        return NULL;
    if (cnt && (!d || !ids)) {
        PyErr_SetString(PyExc_ValueError, "get_batch_ids: null descriptor or id array");
        return NULL;
    }
    t2i_get_desc* g = (t2i_get_desc*)d;
    const t2i_id* src = (const t2i_id*)ids;
    for (uint32_t i = 0; i < cnt; ++i) g[i].id = src[i];
    return PyLong_FromLong(t2i_get_batch((t2i_store*)h, g, cnt, (t2i_status*)per, s));
}

/* free(store, ids, n) -> status (t2i_free) */
static PyObject* py_free(PyObject* self, PyObject* const* args, Py_ssize_t n) {
    void *h, *ids;
    uint32_t cnt;
    (void)self;
    if (!nargs_ok(n, 3, "free") || !arg_ptr(args, 0, &h) || !arg_ptr(args, 1, &ids) || !arg_u32(args, 2, &cnt))
        return NULL;
    return PyLong_FromLong(t2i_free((t2i_store*)h, (const t2i_id*)ids, cnt));
}

static PyMethodDef methods[] = {
    {"put_batch", (PyCFunction)(void (*)(void))py_put_batch, METH_FASTCALL,
     "put_batch(store, descs, n, out_ids, stream) -> status: t2i_put_batch"},
    {"get_batch", (PyCFunction)(void (*)(void))py_get_batch, METH_FASTCALL,
     "get_batch(store, descs, n, per_item, stream) -> status: t2i_get_batch"},
    {"get_batch_ids", (PyCFunction)(void (*)(void))py_get_batch_ids, METH_FASTCALL,
     "get_batch_ids(store, descs, n, ids, per_item, stream) -> status: sets the descriptors' ids, then "
     "t2i_get_batch"},
    {"free", (PyCFunction)(void (*)(void))py_free, METH_FASTCALL, "free(store, ids, n) -> status: t2i_free"},
    {NULL, NULL, 0, NULL}};

static struct PyModuleDef module = {PyModuleDef_HEAD_INIT, "_pycall",
                                    "CPython entry points for the store's per-request calls", -1, methods,
                                    NULL, NULL, NULL, NULL};

PyMODINIT_FUNC PyInit__pycall(void) { return PyModule_Create(&module); }
