"""GB300-native masked ring-matmul path of MOSAIC (arxiv 2607.29221).

``mosaic``    ctypes binding of libmosaic.so (include/mosaic.h)
``protocol``  host-side sequencing of Pi_Sec-Linear on one GPU
``workloads`` seeded synthetic inputs and workload shapes
``build``     nvcc build of the library for sm_103a
"""
